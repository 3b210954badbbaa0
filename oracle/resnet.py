"""ResNet-18-shaped PalQuant network on the oracle -- test infrastructure only.

The paper evaluates PalQuant on ResNet-18 (Sec. 5); its network figure (Fig. 3) is
not available, so the network follows this plain reading, built only from the
oracle's own functions:

* stem: 7x7 stride-2 pad-3 full-precision convolution 3 -> G*w1 channels, ReLU, then
  3x3 stride-2 pad-1 max pooling (the first layer stays in full precision, Sec. 5);
* four stages of two basic blocks with per-group widths w_s (G groups each).  A
  block's input is an fp32 tensor X and its codes Q (Eq. 2 with the block's input
  steps):
    conv1  PalQuant 3x3 layer on Q (stride 2 in the first block of stages 2-4),
           ReLU, no permutation, requantised for conv2 (codes only);
    down   where the block changes shape: PalQuant 1x1 layer on Q with the block's
           stride, no ReLU, no permutation, fp32 out;
    conv2  PalQuant 3x3 layer on conv1's codes, + shortcut (down's output, else X)
           before ReLU, then the cyclic permutation of Eq. 6-8; fp32 out (the next
           block's X) and its codes for the next block (from the post-add value with
           the next block's input steps of the destination group);
* global average pooling and a full-precision FC layer (the last layer stays in
  full precision, Sec. 5).

Placement "paper" follows Sec. 4.3 instead: a cyclic shuffle module (Eq. 9-10,
weights "s{k}.csm" [G, c, 1, 1, c]) at the beginning of each stage, on the stage's
input (X, Q): Z = X + Conv1x1(CyclicPermute(Q)), no ReLU, with Z's codes for the
stage's first block; inside the stage no group permutation; the channel shuffle
(kind 2, ShuffleNet's transpose) once per stage (the paper's default), at the end of
the stage's last block, i.e. in that block's conv2 epilogue after the shortcut add
and ReLU; that output is fp32 only (a per-channel scatter of codes would mix groups
with different steps), and the next stage's input codes come from it by the
quantiser with that stage's module input steps.  Steps keys: "s{k}.csm.in" (module
input), "s{k}.csm.w", and the blocks' keys as in the plain placement.

Steps.  calibrate() derives every step from fp32 tensors of one forward pass: a
layer's weight steps from its weights (LSQ init), a block's input steps from X, the
conv1 output steps from conv1's rescaled output.  forward() takes those steps as
given; both sides of a parity test use the same steps.
"""
from __future__ import annotations

import numpy as np

from . import (avgpool_f32, conv2d_f32, cyclic_shuffle_module, epilogue_scales, group_perm, inv_step, layer,
               linear_f32, maxpool_f32, quantize_act, quantize_weights, act_step, weight_step)


def _blocks(params: dict):
    """(name, stride, has_down) of the eight basic blocks, in order."""
    out = []
    for s in range(4):
        for b in range(2):
            name = f"s{s + 1}b{b + 1}"
            out.append((name, 2 if (s > 0 and b == 0) else 1, (name + ".down") in params))
    return out


def calibrate(x: np.ndarray, params: dict, G: int, bits: int, placement: str = "block") -> dict:
    """Steps of every PalQuant layer from one forward pass in fp32 (see module doc)."""
    return _run(x, params, G, bits, None, placement)["steps"]


def forward(x: np.ndarray, params: dict, G: int, bits: int, steps: dict, placement: str = "block") -> dict:
    """Forward pass with the given steps.  Returns every intermediate tensor:
    "stem", "pool", per block "<b>.in_codes", "<b>.mid_codes", "<b>.down" (if any),
    "<b>.out" (fp32), "<b>.out_codes" (not for the last block; placement "paper":
    first blocks of a stage only), "avg", "logits"; placement "paper" also per stage
    "s{k}.csm.in_codes", "s{k}.csm.out" (fp32 Z) and "s{k}.csm.out_codes"."""
    return _run(x, params, G, bits, steps, placement)


def _run(x, params, G, bits, steps, placement="block"):
    if placement not in ("block", "paper"):
        raise ValueError("placement must be 'block' or 'paper'")
    paper = placement == "paper"
    calib = steps is None
    st = {} if calib else steps
    r = {}
    stem = conv2d_f32(x, params["stem"], 2, 3, relu=True)
    X = maxpool_f32(stem, 3, 2, 1)
    r["stem"], r["pool"] = stem, X
    blocks = _blocks(params)
    first_key = "s1.csm.in" if paper else blocks[0][0] + ".in"
    if calib:
        st[first_key] = act_step(X, G, bits)
    Q = quantize_act(X, G, bits, inv_step(st[first_key]))
    dst = group_perm(G, 1, 1)
    src = [(g - 1) % G for g in range(G)]  # the module's conv group g reads input group pi^-1(g)
    for i, (name, stride, has_down) in enumerate(blocks):
        stage, first_in_stage = int(name[1]), name.endswith("b1")
        if paper and first_in_stage:
            # cyclic shuffle module at the beginning of the stage (Eq. 9-10)
            csm = f"s{stage}.csm"
            r[csm + ".in_codes"] = Q
            wc = params[csm]
            if calib:
                st[csm + ".w"] = weight_step(wc, bits)
            wqc = quantize_weights(wc, bits, inv_step(st[csm + ".w"]))
            m_outc, _ = epilogue_scales(st[csm + ".w"], np.asarray(st[csm + ".in"])[src], None, 1.0, 0, 0)
            if calib:
                Z, _ = cyclic_shuffle_module(X, Q, wqc, m_outc, None, 1, False, bits)
                st[name + ".in"] = act_step(Z, G, bits)
            Z, Qz = cyclic_shuffle_module(X, Q, wqc, m_outc, inv_step(st[name + ".in"]), 1, False, bits)
            r[csm + ".out"], r[csm + ".out_codes"] = Z, Qz
            X, Q = Z, Qz
        s_in = st[name + ".in"]
        r[name + ".in_codes"] = Q
        # conv1: codes for conv2
        w1 = params[name + ".conv1"]
        if calib:
            st[name + ".conv1.w"] = weight_step(w1, bits)
        wq1 = quantize_weights(w1, bits, inv_step(st[name + ".conv1.w"]))
        if calib:
            m_out1, _ = epilogue_scales(st[name + ".conv1.w"], s_in, None, 1.0, 0, 0)
            _, y1, _ = layer(Q, wq1, stride, 1, m_out1, None, 0, 0, relu=True, bits_out=bits)
            st[name + ".mid"] = act_step(y1, G, bits)
        m_out1, m_req1 = epilogue_scales(st[name + ".conv1.w"], s_in, st[name + ".mid"], 1.0, 0, 0)
        _, _, Q1 = layer(Q, wq1, stride, 1, m_out1, m_req1, 0, 0, relu=True, bits_out=bits)
        r[name + ".mid_codes"] = Q1
        # shortcut
        if has_down:
            wd = params[name + ".down"]
            if calib:
                st[name + ".down.w"] = weight_step(wd, bits)
            wqd = quantize_weights(wd, bits, inv_step(st[name + ".down.w"]))
            m_outd, _ = epilogue_scales(st[name + ".down.w"], s_in, None, 1.0, 0, 0)
            _, S, _ = layer(Q, wqd, stride, 0, m_outd, None, 0, 0, relu=False, bits_out=bits)
            r[name + ".down"] = S
        else:
            S = X
        # conv2: + shortcut, ReLU, cyclic permutation; fp32 out and the next block's codes
        w2 = params[name + ".conv2"]
        if calib:
            st[name + ".conv2.w"] = weight_step(w2, bits)
        wq2 = quantize_weights(w2, bits, inv_step(st[name + ".conv2.w"]))
        m_out2, _ = epilogue_scales(st[name + ".conv2.w"], st[name + ".mid"], None, 1.0, 1, 1)
        last = i == len(blocks) - 1
        if paper:
            if first_in_stage:
                # no permutation inside the stage: codes for the stage's second block
                nxt = blocks[i + 1][0] + ".in"
                if calib:
                    _, Xn, _ = layer(Q1, wq2, 1, 1, m_out2, None, 0, 0, shortcut=S, relu=True, bits_out=bits)
                    st[nxt] = act_step(Xn, G, bits)
                _, Xn, Qn = layer(Q1, wq2, 1, 1, m_out2, inv_step(st[nxt]), 0, 0, shortcut=S, relu=True,
                                  bits_out=bits)
                r[name + ".out"], r[name + ".out_codes"] = Xn, Qn
            else:
                # the stage's last block: channel shuffle after the add and ReLU, fp32 out;
                # the next stage's input codes from the quantiser
                _, Xn, _ = layer(Q1, wq2, 1, 1, m_out2, None, 2, 0, shortcut=S, relu=True, bits_out=bits)
                r[name + ".out"] = Xn
                Qn = None
                if not last:
                    nk = f"s{stage + 1}.csm.in"
                    if calib:
                        st[nk] = act_step(Xn, G, bits)
                    Qn = quantize_act(Xn, G, bits, inv_step(st[nk]))
            X, Q = Xn, Qn
            continue
        nxt = None if last else blocks[i + 1][0] + ".in"
        if not last and calib:
            _, Xn, _ = layer(Q1, wq2, 1, 1, m_out2, None, 1, 1, shortcut=S, relu=True, bits_out=bits)
            st[nxt] = act_step(Xn, G, bits)
        # the code of source group g lands in group dst[g]: its multiplier is fl(1/s) of that group
        m_req2 = None if last else inv_step(st[nxt])[dst]
        _, Xn, Qn = layer(Q1, wq2, 1, 1, m_out2, m_req2, 1, 1, shortcut=S, relu=True, bits_out=bits)
        r[name + ".out"] = Xn
        if not last:
            r[name + ".out_codes"] = Qn
        X, Q = Xn, Qn
    v = avgpool_f32(X)
    r["avg"] = v
    r["logits"] = linear_f32(v, params["fc"])
    r["steps"] = st
    return r
