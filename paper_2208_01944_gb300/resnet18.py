"""ResNet-18-shaped PalQuant network on one GPU, driven through the C ABI.

The paper evaluates PalQuant on ResNet-18 (Sec. 5): every body convolution becomes a
PalQuant layer with G groups of B-bit codes (Sec. 4.1), a cyclic permutation moves
each block's output groups on (Sec. 4.2, Eq. 6-8), and the first and last layers stay
in full precision (Sec. 5).  The paper's network figure is not available; this driver
takes the following reading:

* stem: 7x7 stride-2 pad-3 fp32 convolution (3 -> G*w_1 channels) + ReLU, then 3x3
  stride-2 pad-1 max pooling (one kernel for 128 stem channels); the pooled tensor
  is quantised once into codes (inside the first conv1, which then reads the pooled
  fp32 and quantises it on load, where that layer allows it);
* four stages of two basic blocks (per-group widths w_1..w_4).  In block (X, Q):
    conv1  PalQuant 3x3 (stride 2 in the first block of stages 2-4), ReLU, no
           permutation, codes out (requantised with conv2's input steps);
    down   (first block of stages 2-4) PalQuant 1x1 with the block's stride on Q,
           no ReLU, no permutation, fp32 out: the shortcut;
    conv2  PalQuant 3x3 on conv1's codes + shortcut (down's output, else X), ReLU,
           cyclic permutation; fp32 out (the next block's X) and, fused in the same
           epilogue, the next block's codes (multiplier fl(1/s) of the destination
           group's input step);
* global average pooling and an fp32 FC layer.

placement="paper" follows Sec. 4.3 instead (weights from
synth.resnet18_inputs(..., cyclic_modules=True)): a cyclic shuffle module (Eq. 9-10,
palquant_cyclic_shuffle_module: 1x1 group convolution of the group-permuted codes +
the fp32 input, no ReLU) at the beginning of each stage, whose codes feed the stage's
first block; no group permutation inside a stage; the channel shuffle (ShuffleNet's
transpose, shuffle kind 2) once per stage, in the epilogue of the stage's last conv2
after the shortcut add and ReLU, with fp32 output only; the next stage's input codes
then come from the quantiser with that stage's module input steps.

Every step runs in the library's kernels; this module only owns buffers, derives
per-layer multipliers through palquant_epilogue_scales and launches the calls on one
stream, with no host synchronisation inside forward() (which can be captured in a
CUDA graph).  Codes between layers are packed FP4 nibbles (PQ_CODES_C32F4, the
block-scaled FP4 tensor-core path) when the codes have at most 2 bits and every
per-group width is a multiple of 64, else one code per byte, channel-blocked
(PQ_CODES_C16); code_format chooses explicitly.  A code tensor is held as
[N, H, W, C] bytes, or [N, H, W, C/2] for FP4 nibbles.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as B


def _out(n: int, k: int, s: int, p: int) -> int:
    return (n + 2 * p - k) // s + 1


class PalQuantResNet18:
    def __init__(self, params: dict, N: int, H: int = 224, W: int = 224, G: int = 2, widths=(64, 128, 256, 512),
                 classes: int = 1000, bits: int = 2, device="cuda:0", stream: torch.cuda.Stream | None = None,
                 code_format: int | None = None, placement: str = "block", keep_stem: bool = False):
        if placement not in ("block", "paper"):
            raise ValueError("placement must be 'block' or 'paper'")
        self.placement = placement
        self.paper = paper = placement == "paper"
        self.dev = torch.device(device)
        self.N, self.H, self.W, self.G, self.bits, self.classes = N, H, W, G, bits, classes
        self.stream = stream or torch.cuda.Stream(device=self.dev)
        if code_format is None:
            f4_ok = bits <= 2 and all(w % 64 == 0 for w in widths)
            code_format = B.PQ_CODES_C32F4 if f4_ok else B.PQ_CODES_C16
        if code_format not in (B.PQ_CODES_C16, B.PQ_CODES_C32F4):
            raise ValueError("code_format must be PQ_CODES_C16 or PQ_CODES_C32F4")
        self.fmt = fmt = code_format
        per_byte = 2 if fmt == B.PQ_CODES_C32F4 else 1  # codes per byte
        f32 = dict(dtype=torch.float32, device=self.dev)
        u8 = dict(dtype=torch.uint8, device=self.dev)
        self.params = params
        C0 = G * widths[0]
        self.Hs, self.Ws = _out(H, 7, 2, 3), _out(W, 7, 2, 3)
        self.Hp, self.Wp = _out(self.Hs, 3, 2, 1), _out(self.Ws, 3, 2, 1)
        self.C0 = C0
        self.w_stem = torch.from_numpy(np.ascontiguousarray(params["stem"])).to(self.dev)
        self.w_fc = torch.from_numpy(np.ascontiguousarray(params["fc"])).to(self.dev)
        # The stem and the max pooling run as one kernel for 128 stem channels (the
        # stem output then stays on chip unless keep_stem asks for it), else as two.
        self.fused_stem = C0 == 128
        self.stem_out = torch.empty((N, self.Hs, self.Ws, C0), **f32) if keep_stem or not self.fused_stem else None
        self.pool = torch.empty((N, self.Hp, self.Wp, C0), **f32)
        self.in_codes = torch.empty((N, self.Hp, self.Wp, C0 // per_byte), **u8)
        self.blocks = []
        self.modules = []  # placement "paper": one cyclic shuffle module per stage
        Hc, Wc, cin = self.Hp, self.Wp, widths[0]
        for s, w in enumerate(widths):
            if paper:
                m = dict(name=f"s{s + 1}.csm", H=Hc, W=Wc, c=cin)
                m["d"] = B.layer_desc(N, Hc, Wc, G, cin, cin, 1, 1, 0, bits, bits, bits, 0, code_format=fmt)
                m["in_codes"] = self.in_codes if s == 0 else torch.empty((N, Hc, Wc, G * cin // per_byte), **u8)
                m["z"] = torch.empty((N, Hc, Wc, G * cin), **f32)
                m["codes"] = torch.empty((N, Hc, Wc, G * cin // per_byte), **u8)
                m["wp"] = torch.empty(B.palquant_packed_weight_bytes(m["d"]), **u8)
                self.modules.append(m)
            for b in range(2):
                name = f"s{s + 1}b{b + 1}"
                stride = 2 if (s > 0 and b == 0) else 1
                Ho, Wo = _out(Hc, 3, stride, 1), _out(Wc, 3, stride, 1)
                blk = dict(name=name, stride=stride, cin=cin, w=w, H=Hc, W=Wc, Ho=Ho, Wo=Wo,
                           down=(name + ".down") in params)
                blk["d1"] = B.layer_desc(N, Hc, Wc, G, cin, w, 3, stride, 1, bits, bits, bits, 1, code_format=fmt)
                blk["d2"] = B.layer_desc(N, Ho, Wo, G, w, w, 3, 1, 1, bits, bits, bits, 1, code_format=fmt)
                if blk["down"]:
                    blk["dd"] = B.layer_desc(N, Hc, Wc, G, cin, w, 1, stride, 0, bits, bits, bits, 0, code_format=fmt)
                    blk["down_out"] = torch.empty((N, Ho, Wo, G * w), **f32)
                blk["mid_codes"] = torch.empty((N, Ho, Wo, G * w // per_byte), **u8)
                blk["out"] = torch.empty((N, Ho, Wo, G * w), **f32)
                blk["out_codes"] = torch.empty((N, Ho, Wo, G * w // per_byte), **u8)
                for key, d in (("wp1", blk["d1"]), ("wp2", blk["d2"])) + ((("wpd", blk["dd"]),) if blk["down"] else ()):
                    blk[key] = torch.empty(B.palquant_packed_weight_bytes(d), **u8)
                self.blocks.append(blk)
                Hc, Wc, cin = Ho, Wo, w
        self.Hl, self.Wl, self.Cl = Hc, Wc, G * cin
        self.avg = torch.empty((N, self.Cl), **f32)
        self.logits = torch.empty((N, classes), **f32)
        self.no_shuffle = B.shuffle(0, 0)
        self.cyclic = B.shuffle(1, 1)
        self.channel_shuffle = B.shuffle(2, 0)
        self.ones = np.ones(G, dtype=np.float32)
        self.steps = None
        self.graph = None
        self.fuse_input = False  # set by set_steps()

    # --------------------------------------------------------------- set-up
    def _inv(self, s, shuf=None):
        """fl(1/s[dst(g)]) per source group g, computed by the library in double."""
        return B.palquant_epilogue_scales(self.G, self.ones, self.ones, 1.0, s, shuf or self.no_shuffle)[1]

    def _act_steps(self, t: torch.Tensor, Cg: int) -> np.ndarray:
        N, H, W, C = t.shape
        nbytes = B.palquant_act_steps_scratch_bytes(N * H * W, self.G)
        scratch = torch.empty(nbytes, dtype=torch.uint8, device=self.dev)
        return B.palquant_act_steps(t, N, H, W, self.G, Cg, self.bits, scratch, nbytes, stream=self.stream)

    def calibrate(self, x_dev: torch.Tensor) -> dict:
        """Steps of every PalQuant layer from one fp32 pass over x (LSQ initialisation:
        weights from their own values, activations from the tensor entering the layer)."""
        if self.paper:
            return self._calibrate_paper(x_dev)
        G, bits, st = self.G, self.bits, {}
        s = self.stream
        self._stem(x_dev)
        first = self.blocks[0]["name"]
        st[first + ".in"] = self._act_steps(self.pool, self.C0 // G)
        for i, blk in enumerate(self.blocks):
            n = blk["name"]
            st[n + ".conv1.w"] = B.palquant_weight_steps(self.params[n + ".conv1"], blk["d1"])
            st[n + ".conv2.w"] = B.palquant_weight_steps(self.params[n + ".conv2"], blk["d2"])
            if blk["down"]:
                st[n + ".down.w"] = B.palquant_weight_steps(self.params[n + ".down"], blk["dd"])
        # activation steps layer by layer: each needs the previous layers' codes
        self.steps = st
        for i, blk in enumerate(self.blocks):
            n = blk["name"]
            self._pack(blk, st)
            self._scales(blk, st)
            if i == 0:
                B.palquant_quantize_act(self.pool, self.in_codes, self.N, self.Hp, self.Wp, G, self.C0 // G, bits,
                                        self._inv(st[n + ".in"]), code_format=self.fmt, stream=s)
            q_in = self.in_codes if i == 0 else self.blocks[i - 1]["out_codes"]
            m_out1, _ = B.palquant_epilogue_scales(G, st[n + ".conv1.w"], st[n + ".in"], 1.0, None, self.no_shuffle)
            y1 = torch.empty((self.N, blk["Ho"], blk["Wo"], G * blk["w"]), dtype=torch.float32, device=self.dev)
            B.palquant_layer_fused(q_in, blk["wp1"], blk["d1"], m_out1, None, self.no_shuffle, None, None, y1, None,
                                   stream=s)
            st[n + ".mid"] = self._act_steps(y1, blk["w"])
            del y1
            self._scales(blk, st)
            self._block_front(blk, q_in)
            if i + 1 < len(self.blocks):
                self._conv2(blk, None)  # fp32 output only
                nxt = self.blocks[i + 1]["name"] + ".in"
                st[nxt] = self._act_steps(blk["out"], blk["w"])
                # the next block's codes, as forward() fuses them into conv2
                self._conv2(blk, self._inv(st[nxt], self.cyclic))
        self.set_steps(st)
        return st

    def _calibrate_paper(self, x_dev: torch.Tensor) -> dict:
        """calibrate() for placement "paper", in the order the oracle network takes."""
        G, bits, st, s = self.G, self.bits, {}, self.stream
        self._stem(x_dev)
        st["s1.csm.in"] = self._act_steps(self.pool, self.C0 // G)
        for blk in self.blocks:
            n = blk["name"]
            st[n + ".conv1.w"] = B.palquant_weight_steps(self.params[n + ".conv1"], blk["d1"])
            st[n + ".conv2.w"] = B.palquant_weight_steps(self.params[n + ".conv2"], blk["d2"])
            if blk["down"]:
                st[n + ".down.w"] = B.palquant_weight_steps(self.params[n + ".down"], blk["dd"])
        for m in self.modules:
            st[m["name"] + ".w"] = B.palquant_weight_steps(self.params[m["name"]], m["d"])
        self.steps = st
        B.palquant_quantize_act(self.pool, self.in_codes, self.N, self.Hp, self.Wp, G, self.C0 // G, bits,
                                self._inv(st["s1.csm.in"]), code_format=self.fmt, stream=s)
        X = self.pool
        for k, m in enumerate(self.modules):
            b1, b2 = self.blocks[2 * k], self.blocks[2 * k + 1]
            self._pack_module(m, st)
            B.palquant_cyclic_shuffle_module(m["in_codes"], m["wp"], m["d"], m["m_out"], None, 1, X, m["z"], None,
                                             stream=s)
            st[b1["name"] + ".in"] = self._act_steps(m["z"], m["c"])
            m["m_req"] = self._inv(st[b1["name"] + ".in"])
            B.palquant_cyclic_shuffle_module(m["in_codes"], m["wp"], m["d"], m["m_out"], m["m_req"], 1, X, m["z"],
                                             m["codes"], stream=s)
            for blk, q_in in ((b1, m["codes"]), (b2, b1["out_codes"])):
                n = blk["name"]
                self._pack(blk, st)
                m_out1, _ = B.palquant_epilogue_scales(G, st[n + ".conv1.w"], st[n + ".in"], 1.0, None, self.no_shuffle)
                y1 = torch.empty((self.N, blk["Ho"], blk["Wo"], G * blk["w"]), dtype=torch.float32, device=self.dev)
                B.palquant_layer_fused(q_in, blk["wp1"], blk["d1"], m_out1, None, self.no_shuffle, None, None, y1, None,
                                       stream=s)
                st[n + ".mid"] = self._act_steps(y1, blk["w"])
                del y1
                self._scales(blk, st)
                self._block_front(blk, q_in)
                if blk is b1:
                    sc = b1["down_out"] if b1["down"] else m["z"]
                    self._conv2_paper(b1, sc, None, False)
                    st[b2["name"] + ".in"] = self._act_steps(b1["out"], b1["w"])
                    self._conv2_paper(b1, sc, self._inv(st[b2["name"] + ".in"]), False)
                else:
                    self._conv2_paper(b2, b1["out"], None, True)
                    if k + 1 < len(self.modules):
                        nxt = self.modules[k + 1]
                        st[nxt["name"] + ".in"] = self._act_steps(b2["out"], b2["w"])
                        B.palquant_quantize_act(b2["out"], nxt["in_codes"], self.N, b2["Ho"], b2["Wo"], G, b2["w"],
                                                bits, self._inv(st[nxt["name"] + ".in"]), code_format=self.fmt,
                                                stream=s)
            X = b2["out"]
        self.set_steps(st)
        return st

    def _pack_module(self, m, st):
        """Pack a stage's module weights; its multiplier m_out[g] = fl(s_w[g] s_in[pi^-1(g)])
        (conv group g reads the permuted input group)."""
        n, G = m["name"], self.G
        B.palquant_pack_weights(self.params[n], m["d"], self._inv(st[n + ".w"]), m["wp"], m["wp"].numel(),
                                stream=self.stream)
        src = [(g - 1) % G for g in range(G)]
        s_in = np.asarray(st[n + ".in"], dtype=np.float32)[src]
        m["m_out"] = B.palquant_epilogue_scales(G, st[n + ".w"], s_in, 1.0, None, self.no_shuffle)[0]

    def _conv2_paper(self, blk, shortcut, m_req2, last):
        """conv2 of placement "paper": no permutation and the codes of the stage's second
        block, or (the stage's last block) the channel shuffle and fp32 out only."""
        B.palquant_layer_fused(blk["mid_codes"], blk["wp2"], blk["d2"], blk["m_out2"], None if last else m_req2,
                               self.channel_shuffle if last else self.no_shuffle, shortcut, None, blk["out"],
                               None if (last or m_req2 is None) else blk["out_codes"], stream=self.stream)

    def _pack(self, blk, st):
        """Quantise and pack the block's weights with their steps (synchronous)."""
        n = blk["name"]
        for key, d, wname in (("wp1", blk["d1"], ".conv1"), ("wp2", blk["d2"], ".conv2")) + \
                ((("wpd", blk["dd"], ".down"),) if blk["down"] else ()):
            B.palquant_pack_weights(self.params[n + wname], d, self._inv(st[n + wname + ".w"]), blk[key],
                                    blk[key].numel(), stream=self.stream)

    def _scales(self, blk, st):
        """Epilogue multipliers of the block's layers from the steps known so far."""
        n, G = blk["name"], self.G
        blk["m_out1"], blk["m_req1"] = B.palquant_epilogue_scales(G, st[n + ".conv1.w"], st[n + ".in"], 1.0,
                                                                  st.get(n + ".mid"), self.no_shuffle)
        if blk["down"]:
            blk["m_outd"], _ = B.palquant_epilogue_scales(G, st[n + ".down.w"], st[n + ".in"], 1.0, None,
                                                          self.no_shuffle)
        if n + ".mid" in st:
            blk["m_out2"], _ = B.palquant_epilogue_scales(G, st[n + ".conv2.w"], st[n + ".mid"], 1.0, None, self.cyclic)

    def set_steps(self, steps: dict):
        """Pack every layer's weights and derive the epilogue multipliers from `steps`."""
        self.steps = dict(steps)
        if self.paper:
            for k, m in enumerate(self.modules):
                self._pack_module(m, self.steps)
                m["inv_in"] = self._inv(self.steps[m["name"] + ".in"])
                m["m_req"] = self._inv(self.steps[self.blocks[2 * k]["name"] + ".in"])
            for i, blk in enumerate(self.blocks):
                self._pack(blk, self.steps)
                self._scales(blk, self.steps)
                first = blk["name"].endswith("b1")
                blk["m_req2"] = self._inv(self.steps[self.blocks[i + 1]["name"] + ".in"]) if first else None
            self.inv_in = self.modules[0]["inv_in"]
            self.stream.synchronize()
            self.graph = None
            return
        for i, blk in enumerate(self.blocks):
            self._pack(blk, self.steps)
            self._scales(blk, self.steps)
            nxt = self.blocks[i + 1]["name"] + ".in" if i + 1 < len(self.blocks) else None
            # conv2's codes land in group dst(g) of the next block: multiplier fl(1/s_next[dst(g)])
            blk["m_req2"] = None if nxt is None else self._inv(self.steps[nxt], self.cyclic)
        self.inv_in = self._inv(self.steps[self.blocks[0]["name"] + ".in"])
        # The input quantiser runs inside the first conv1 (quantise-on-load: the fp32
        # pooled tensor in, its codes only in shared memory) where that layer can take
        # it: stride 1 and no downsample reading the input codes.  A shape the fused
        # call rejects keeps the separate quantiser.
        b0 = self.blocks[0]
        self.fuse_input = False
        if not b0["down"] and b0["stride"] == 1:
            try:
                B.palquant_quantize_layer_fused(self.pool, self.inv_in, b0["wp1"], b0["d1"], b0["m_out1"],
                                                b0["m_req1"], self.no_shuffle, None, None, None, b0["mid_codes"],
                                                stream=self.stream)
                self.fuse_input = True
            except B.PalquantError as e:
                if e.status not in (B.PQ_EUNSUPPORTED, B.PQ_EINVAL):
                    raise
        self.stream.synchronize()
        self.graph = None

    # --------------------------------------------------------------- forward
    def _stem(self, x_dev):
        s = self.stream
        if self.fused_stem:
            B.palquant_stem_pool_f32(x_dev, self.w_stem, self.stem_out, self.pool, self.N, self.H, self.W, self.C0,
                                     stream=s)
            return
        B.palquant_conv2d_f32(x_dev, self.w_stem, self.stem_out, self.N, self.H, self.W, 3, self.C0, 7, 2, 3, relu=True,
                              stream=s)
        B.palquant_maxpool2d_f32(self.stem_out, self.pool, self.N, self.Hs, self.Ws, self.C0, 3, 2, 1, stream=s)

    def _block_front(self, blk, q_in):
        s = self.stream
        B.palquant_layer_fused(q_in, blk["wp1"], blk["d1"], blk["m_out1"], blk["m_req1"], self.no_shuffle, None, None,
                               None, blk["mid_codes"], stream=s)
        if blk["down"]:
            B.palquant_layer_fused(q_in, blk["wpd"], blk["dd"], blk["m_outd"], None, self.no_shuffle, None, None,
                                   blk["down_out"], None, stream=s)

    def _conv2(self, blk, m_req2):
        i = self.blocks.index(blk)
        shortcut = blk["down_out"] if blk["down"] else (self.pool if i == 0 else self.blocks[i - 1]["out"])
        B.palquant_layer_fused(blk["mid_codes"], blk["wp2"], blk["d2"], blk["m_out2"], m_req2, self.cyclic, shortcut,
                               None, blk["out"], None if m_req2 is None else blk["out_codes"], stream=self.stream)

    def forward(self, x_dev: torch.Tensor, marks: list | None = None) -> torch.Tensor:
        """Logits [N, classes] for images x_dev (NHWC fp32 [N, H, W, 3] on the device);
        asynchronous on self.stream.  With `marks`, a CUDA event recorded on the stream
        after each stage is appended as (stage name, event)."""
        if self.steps is None:
            raise RuntimeError("calibrate() or set_steps() first")
        s = self.stream

        def mark(name):
            if marks is not None:
                ev = torch.cuda.Event(enable_timing=True)
                ev.record(s)
                marks.append((name, ev))

        mark("start")
        self._stem(x_dev)
        mark("stem conv + max pooling (fp32)")
        fused_in = self.fuse_input and not self.paper
        if not fused_in:
            B.palquant_quantize_act(self.pool, self.in_codes, self.N, self.Hp, self.Wp, self.G, self.C0 // self.G,
                                    self.bits, self.inv_in, code_format=self.fmt, stream=s)
            mark("input quantiser")
        if self.paper:
            X = self.pool
            for k, m in enumerate(self.modules):
                b1, b2 = self.blocks[2 * k], self.blocks[2 * k + 1]
                B.palquant_cyclic_shuffle_module(m["in_codes"], m["wp"], m["d"], m["m_out"], m["m_req"], 1, X, m["z"],
                                                 m["codes"], stream=s)
                mark(m["name"] + " cyclic shuffle module")
                self._block_front(b1, m["codes"])
                mark(b1["name"] + " conv1" + (" + down" if b1["down"] else ""))
                self._conv2_paper(b1, b1["down_out"] if b1["down"] else m["z"], b1["m_req2"], False)
                mark(b1["name"] + " conv2")
                self._block_front(b2, b1["out_codes"])
                mark(b2["name"] + " conv1")
                self._conv2_paper(b2, b1["out"], None, True)
                mark(b2["name"] + " conv2 + channel shuffle")
                if k + 1 < len(self.modules):
                    nxt = self.modules[k + 1]
                    B.palquant_quantize_act(b2["out"], nxt["in_codes"], self.N, b2["Ho"], b2["Wo"], self.G, b2["w"],
                                            self.bits, nxt["inv_in"], code_format=self.fmt, stream=s)
                    mark(nxt["name"] + " input quantiser")
                X = b2["out"]
        else:
            for i, blk in enumerate(self.blocks):
                if i == 0 and fused_in:
                    B.palquant_quantize_layer_fused(self.pool, self.inv_in, blk["wp1"], blk["d1"], blk["m_out1"],
                                                    blk["m_req1"], self.no_shuffle, None, None, None,
                                                    blk["mid_codes"], stream=s)
                    mark(blk["name"] + " conv1 (input quantiser fused)")
                else:
                    q_in = self.in_codes if i == 0 else self.blocks[i - 1]["out_codes"]
                    self._block_front(blk, q_in)
                    mark(blk["name"] + " conv1" + (" + down" if blk["down"] else ""))
                self._conv2(blk, blk["m_req2"])
                mark(blk["name"] + " conv2")
        last = self.blocks[-1]["out"]
        B.palquant_avgpool_f32(last, self.avg, self.N, self.Hl, self.Wl, self.Cl, stream=s)
        B.palquant_linear_f32(self.avg, self.w_fc, self.logits, self.N, self.Cl, self.classes, stream=s)
        mark("average pooling + FC (fp32)")
        return self.logits

    def capture(self, x_dev: torch.Tensor):
        """Capture forward(x_dev) into a CUDA graph (replayed by replay())."""
        self.forward(x_dev)  # warm-up outside capture (first-call set-up in the library)
        self.stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=self.stream):
            self.forward(x_dev)
        self.graph = g
        return g

    def replay(self, graph=None):
        """Replay a captured forward on self.stream (the last capture by default)."""
        with torch.cuda.stream(self.stream):
            (graph or self.graph).replay()
        return self.logits

    def launches_per_forward(self) -> int:
        """Kernels one forward launches: the stem with its max pooling (one kernel for
        128 stem channels, else two), quantiser, per block conv1 (+ down) + conv2,
        average pooling, FC."""
        n = (2 if self.fused_stem else 3) + sum(3 if b["down"] else 2 for b in self.blocks) + 2
        if self.fuse_input and not self.paper:
            n -= 1  # the quantiser runs inside the first conv1
        if self.paper:
            n += len(self.modules) + len(self.modules) - 1  # a module per stage, a quantiser per stage boundary
        return n

    def body_int_ops(self) -> int:
        """Integer operations (2 per MAC) of the PalQuant layers of one forward."""
        G, N, ops = self.G, self.N, 0
        for b in self.blocks:
            ops += 2 * N * b["Ho"] * b["Wo"] * G * b["w"] * 9 * b["cin"]
            ops += 2 * N * b["Ho"] * b["Wo"] * G * b["w"] * 9 * b["w"]
            if b["down"]:
                ops += 2 * N * b["Ho"] * b["Wo"] * G * b["w"] * b["cin"]
        for m in self.modules:
            ops += 2 * N * m["H"] * m["W"] * G * m["c"] * m["c"]
        return ops
