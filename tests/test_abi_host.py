"""The C-ABI library on the host (no GPU): exported symbols, planner invariants,
weight packing, host-side set-up against the oracle, and argument validation."""
import os
import re

import numpy as np
import pytest
import torch

import oracle
from paper_2208_01944_gb300 import synth, workloads

B = pytest.importorskip("paper_2208_01944_gb300.binding", reason="libpalquant.so not built")

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "palquant.h")


def _desc(c, **kw):
    args = dict(N=c.N, H=c.H, W=c.W, G=c.G, Cin_g=c.Cin_g, Cout_g=c.Cout_g, k=c.k, stride=c.stride, pad=c.pad,
                bits_a=c.bits_a, bits_w=c.bits_w, bits_out=c.bits_out)
    args.update(kw)
    return B.layer_desc(**args)


def test_every_declared_symbol_is_exported():
    decls = set(re.findall(r"\b(palquant_\w+)\s*\(", open(HEADER).read()))
    assert decls == set(B.EXPORTS)
    for name in decls:
        assert hasattr(B.lib, name), name
    assert B.palquant_version() >= 100
    assert B.strerror(B.PQ_ETIMEOUT) == "in-kernel wait timed out"


def test_raw_code_byte_is_e4m3_of_scaled_code():
    """A code byte v <= 15 is the FP8 E4M3 encoding of v * 2^-9 (checked with torch's fp8 type)."""
    v = torch.arange(16, dtype=torch.uint8)
    as_fp8 = v.view(torch.float8_e4m3fn).to(torch.float64)
    assert torch.equal(as_fp8 * 512.0, v.to(torch.float64))


ALL_LAYERS = list(workloads.BENCH_CONFIGS.values()) + [c for _, _, c in workloads.resnet18_layers()]


@pytest.mark.parametrize("c", ALL_LAYERS, ids=lambda c: f"{c.H}x{c.W}k{c.k}s{c.stride}G{c.G}c{c.Cin_g}-{c.Cout_g}")
def test_plan_invariants(c):
    plan = B.palquant_conv_plan(_desc(c))
    assert plan.supported == 1
    assert plan.smem_bytes + 1024 <= 227 * 1024
    assert plan.n_block * plan.n_blocks == c.Cout_g and plan.n_block % 16 == 0 and 16 <= plan.n_block <= 256
    assert plan.k_chunk * plan.k_blocks == c.Cin_g and plan.k_chunk % 32 == 0
    assert plan.taps == c.k * c.k
    rows = plan.m_tiles * 128
    if plan.mode == 1:
        assert plan.rows_per_tile * plan.tile_pitch <= rows
        tiles_per_img = -(-c.Ho // plan.rows_per_tile)
        assert plan.tiles == c.N * tiles_per_img
        assert plan.tile_pitch >= c.Wo
    else:
        assert plan.tiles == c.N * -(-(c.Ho * c.Wo) // rows)  # flat tiles stay inside one image
    assert plan.work_items == plan.tiles * c.G * plan.n_blocks
    assert plan.acc_stages * plan.m_tiles * plan.n_block <= 512


def test_plan_weight_residency():
    """A (group, output block) unit's packed weights stay in shared memory only up to
    160 KB; the 3x3 layers of 128x28x28 with 4 groups of 128 (147 KB a unit) keep
    theirs, the 2-group ones (590 KB at 256 columns) stream them."""
    for c in ALL_LAYERS:
        plan = B.palquant_conv_plan(_desc(c))
        unit_bytes = c.k * c.k * c.Cin_g * plan.n_block
        if unit_bytes > 160 * 1024:
            assert plan.weights_resident == 0, c
    for name in ("config3_1", "config3_4"):
        c = workloads.BENCH_CONFIGS[name]
        plan = B.palquant_conv_plan(_desc(c))
        assert (c.G, c.Cin_g, plan.n_block, plan.weights_resident) == (4, 128, 128, 1)
    plan = B.palquant_conv_plan(_desc(workloads.BENCH_CONFIGS["config3_0"]))
    assert plan.weights_resident == 0


@pytest.mark.parametrize("shape", [(2, 48, 3, 64, 4), (4, 96, 1, 96, 2), (1, 272, 3, 32, 2), (3, 64, 3, 128, 4)])
def test_pack_unpack_roundtrip_and_fp8_encoding(shape):
    G, Co, k, Ci, bits = shape
    d = B.layer_desc(1, 8, 8, G, Ci, Co, k, 1, k // 2, bits, bits, bits)
    gen = synth.generator(sum(shape))
    wq = synth.random_codes((G, Co, k, k, Ci), bits, gen, signed=True)
    packed = B.palquant_pack_weight_codes_host(wq, d)
    assert packed.size == wq.size
    assert np.array_equal(B.palquant_unpack_weight_codes_host(packed, d), wq)
    # The packed bytes are the FP8 E4M3 encodings of the codes (as a multiset per group
    # they must equal torch's encoding of the same integers).
    fp8 = torch.from_numpy(wq.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(np.sort(packed), np.sort(fp8.ravel()))


def test_pack_rejects_out_of_range_codes():
    d = B.layer_desc(1, 4, 4, 1, 32, 16, 1, 1, 0, 2, 2, 2)
    wq = np.zeros((1, 16, 1, 1, 32), dtype=np.int8)
    wq[0, 3, 0, 0, 5] = 2  # outside [-2, 1] for 2-bit codes
    with pytest.raises(B.PalquantError) as e:
        B.palquant_pack_weight_codes_host(wq, d)
    assert e.value.status == B.PQ_EINVAL


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_weight_quantisation_matches_oracle(bits):
    G, Co, k, Ci = 3, 32, 3, 64
    gen = synth.generator(40 + bits)
    w = synth.he_weights(G, Co, k, k, Ci, gen)
    d = B.layer_desc(1, 6, 6, G, Ci, Co, k, 1, 1, 2, bits, 2)
    s_w = B.palquant_weight_steps(w, d)
    assert np.array_equal(s_w, oracle.weight_step(w, bits))
    inv = oracle.inv_step(s_w)
    packed = B.palquant_pack_weights_host(w, d, inv)
    assert np.array_equal(B.palquant_unpack_weight_codes_host(packed, d), oracle.quantize_weights(w, bits, inv))


def test_weight_quantisation_ties_and_clamp():
    d = B.layer_desc(1, 4, 4, 1, 32, 16, 1, 1, 0, 2, 2, 2)
    w = np.zeros((1, 16, 1, 1, 32), dtype=np.float32)
    w[0, 0, 0, 0, :6] = [0.5, 1.5, -0.5, -1.5, 9.0, -9.0]
    packed = B.palquant_pack_weights_host(w, d, [1.0])
    wq = B.palquant_unpack_weight_codes_host(packed, d)
    assert list(wq[0, 0, 0, 0, :6]) == [0, 1, 0, -2, 1, -2]


@pytest.mark.parametrize("kind,shift,perm", [(0, 0, None), (1, 1, None), (1, -1, None), (3, 0, [2, 0, 3, 1])])
def test_epilogue_scales_match_oracle(kind, shift, perm):
    gen = synth.generator(7)
    s_w = synth.half_normal((4,), gen) + 0.1
    s_a = synth.half_normal((4,), gen) + 0.1
    s_n = synth.half_normal((4,), gen) + 0.1
    mo, mr = B.palquant_epilogue_scales(4, s_w, s_a, 1.25, s_n, B.shuffle(kind, shift, perm))
    ro, rr = oracle.epilogue_scales(s_w, s_a, s_n, 1.25, kind, shift, perm)
    assert np.array_equal(mo, ro) and np.array_equal(mr, rr)


def test_invalid_arguments_rejected_before_launch():
    good = B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1)
    bad_descs = [
        B.layer_desc(1, 0, 8, 2, 32, 32, 3, 1, 1),       # H = 0
        B.layer_desc(1, 8, 8, 0, 32, 32, 3, 1, 1),       # G = 0
        B.layer_desc(1, 8, 8, 2, 32, 32, 3, 0, 1),       # stride 0
        B.layer_desc(1, 2, 2, 2, 32, 32, 5, 1, 0),       # output would be empty
        B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, bits_a=9),
        B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, flags=2),    # unknown flag bit
        B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, flags=-1),
    ]
    for d in bad_descs:
        with pytest.raises(B.PalquantError) as e:
            B.palquant_layer_fused(16, 16, d, [1.0] * 2, [1.0] * 2, acc_out_dev=16)
        assert e.value.status == B.PQ_EINVAL
    # the inputs-ready promise is a valid flag: planning accepts it and plans the same tiles
    ready = B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, code_format=B.PQ_CODES_C16, flags=B.PQ_LAYER_INPUTS_READY)
    plain = B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, code_format=B.PQ_CODES_C16)
    assert B.palquant_conv_plan(ready).as_dict() == B.palquant_conv_plan(plain).as_dict()
    # no output requested
    with pytest.raises(B.PalquantError) as e:
        B.palquant_layer_fused(16, 16, good, [1.0] * 2, [1.0] * 2)
    assert e.value.status == B.PQ_EINVAL
    # codes requested without requantisation multipliers
    with pytest.raises(B.PalquantError) as e:
        B.palquant_layer_fused(16, 16, good, [1.0] * 2, None, q_out_dev=16)
    assert e.value.status == B.PQ_EINVAL
    # misaligned device pointer
    with pytest.raises(B.PalquantError) as e:
        B.palquant_layer_fused(17, 16, good, [1.0] * 2, [1.0] * 2, acc_out_dev=16)
    assert e.value.status == B.PQ_EINVAL
    # not a permutation
    with pytest.raises(B.PalquantError) as e:
        B.palquant_layer_fused(16, 16, good, [1.0] * 2, [1.0] * 2, shuf=B.shuffle(3, 0, [1, 1]), acc_out_dev=16)
    assert e.value.status == B.PQ_EINVAL


def test_unsupported_shapes_reported():
    for d in [B.layer_desc(1, 8, 8, 2, 24, 32, 3, 1, 1),          # Cin_g not a multiple of 32
              B.layer_desc(1, 8, 8, 2, 32, 24, 3, 1, 1),          # Cout_g not a multiple of 16
              B.layer_desc(1, 8, 8, 2, 32, 32, 3, 3, 1),          # stride 3
              B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, bits_a=6)]:  # codes beyond the exact FP8 range
        assert B.palquant_conv_plan(d).supported == 0
        assert B.palquant_packed_weight_bytes(d) == 0
        with pytest.raises(B.PalquantError) as e:
            B.palquant_layer_fused(16, 16, d, [1.0] * 2, [1.0] * 2, acc_out_dev=16)
        assert e.value.status == B.PQ_EUNSUPPORTED


@pytest.mark.parametrize("M,Bb", [(4, 2), (3, 2), (4, 1)])  # shifted values within int8 for the unpacker
def test_bitsplit_weight_blocks_are_shifted_slices(M, Bb):
    """Eq. 4's weight side: block (i, j) of the decomposed weights is 2^((i+j)B) W_j,
    W_j the oracle's slices of the M-bit codes."""
    d = B.layer_desc(1, 8, 8, 1, 32, 16, 3, 1, 1, M, M, 2)
    gen = synth.generator(M * 3 + Bb)
    wq = synth.random_codes((1, 16, 3, 3, 32), M, gen, signed=True)
    B_bits = Bb
    t = B.palquant_bitsplit_desc(d, B_bits)
    Ga = Gw = -(-M // B_bits)
    # each activation slice once (Ga channel blocks), Gw weight slices per tap
    assert t.Cin_g == 32 * Ga and t.wslices == Gw and t.bits_a == B_bits
    packed = B.palquant_bitsplit_pack_weight_codes_host(wq, d, B_bits)
    vals = B.palquant_unpack_weight_codes_host(packed, t).astype(np.int64)  # [1,16,3,3,Gw,Ga*32]
    assert vals.shape == (1, 16, 3, 3, Gw, Ga * 32)
    ws = oracle.bit_slices_weights(wq, M, B_bits)
    for i in range(Ga):
        for j in range(Gw):
            blk = vals[..., j, i * 32:(i + 1) * 32]
            assert np.array_equal(blk, ws[j].astype(np.int64) << ((i + j) * B_bits))


def test_bitsplit_desc_clears_inputs_ready():
    """The decomposed convolution reads the slices the kernel before it writes, so the
    caller's inputs-ready promise does not carry over to it."""
    d = B.layer_desc(2, 8, 8, 1, 32, 32, 3, 1, 1, bits_a=4, bits_w=4, bits_out=4, code_format=B.PQ_CODES_C16,
                     flags=B.PQ_LAYER_INPUTS_READY)
    t = B.palquant_bitsplit_desc(d, 2)
    assert t.flags == 0 and t.Cin_g == 32 * 2 and t.wslices == 2 and t.bits_a == 2


def test_bitsplit_unsupported_shapes():
    # 6-bit on 2-bit hardware: shifted slices reach 3 * 2^8, beyond exact E4M3
    d = B.layer_desc(1, 8, 8, 1, 32, 16, 3, 1, 1, 6, 6, 2)
    with pytest.raises(B.PalquantError) as e:
        B.palquant_bitsplit_desc(d, 2)
    assert e.value.status == B.PQ_EUNSUPPORTED
    assert B.palquant_bitsplit_scratch_bytes(d, 2) == 0
    with pytest.raises(B.PalquantError) as e:
        B.palquant_bitsplit_desc(B.layer_desc(1, 8, 8, 1, 32, 16, 3, 1, 1, 4, 4, 2), 5)
    assert e.value.status == B.PQ_EINVAL


def test_packed_codes_layout_rules():
    """Packed 2-bit codes: 2-bit codes only, stride 1, rows of whole 16-byte multiples."""
    P2 = B.PQ_CODES_C16P2
    ok = B.palquant_conv_plan(B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=P2))
    assert ok.supported == 1
    for d in [B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 4, 4, 4, code_format=P2),   # 4-bit codes
              B.layer_desc(1, 8, 8, 2, 32, 32, 3, 2, 1, 2, 2, 2, code_format=P2),   # stride 2
              B.layer_desc(1, 8, 10, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=P2),  # W % 4 != 0
              B.layer_desc(1, 3, 3, 2, 32, 32, 1, 1, 0, 2, 2, 2, code_format=P2)]:  # 1x1, H W % 4 != 0
        assert B.palquant_conv_plan(d).supported == 0
    # a per-channel scatter cannot write packed codes
    d = B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=P2)
    with pytest.raises(B.PalquantError) as e:
        B.palquant_layer_fused(16, 16, d, [1.0] * 2, [1.0] * 2, shuf=B.shuffle(2, 0), q_out_dev=16)
    assert e.value.status == B.PQ_EUNSUPPORTED


def test_packed_code_helpers_roundtrip():
    from layer_cases import c16p2_to_nhwc, from_format, to_format

    gen = synth.generator(77)
    q = synth.random_codes((2, 3, 4, 32), 2, gen)
    raw = to_format(q, 3)
    assert raw.size == q.size // 4
    assert np.array_equal(c16p2_to_nhwc(raw, 2, 3, 4, 32), q)
    assert np.array_equal(from_format(to_format(q, 2), 2, 2, 3, 4, 32), q)
    # code of channel c at bits 2 (c % 16) of its block's little-endian word
    one = np.zeros((1, 1, 1, 16), np.uint8)
    one[0, 0, 0, 5] = 3
    assert int(to_format(one, 3).view(np.uint32)[0]) == 3 << 10


@pytest.mark.parametrize("bits", [2, 3])
def test_odd_level_weights_match_oracle(bits):
    gen = synth.generator(bits + 60)
    G, Co, k, Ci = 2, 32, 3, 64
    w = synth.he_weights(G, Co, k, k, Ci, gen)
    u = (2.0 * np.abs(w).reshape(G, -1).mean(axis=1)).astype(np.float32)
    d = B.layer_desc(1, 6, 6, G, Ci, Co, k, 1, 1, 2, bits, 2)
    packed = B.palquant_pack_weights_odd_host(w, d, u)
    assert np.array_equal(B.palquant_unpack_weight_codes_host(packed, d), oracle.quantize_weights_odd(w, bits, u))


# --------------------------------------------- packed FP4 codes (format 4)
def _e2m1_value(nib):
    """E2M1 by its definition: sign bit 3, exponent bits 2-1 (bias 1), mantissa bit 0;
    exponent 0 is subnormal (m * 0.5)."""
    nib = np.asarray(nib, dtype=np.int64)
    s = np.where(nib & 8, -1.0, 1.0)
    e, m = (nib >> 1) & 3, nib & 1
    mag = np.where(e == 0, m * 0.5, (1.0 + m / 2.0) * 2.0 ** (e - 1))
    return s * mag


def test_fp4_nibble_of_code_is_e2m1_of_half_code():
    """An activation code v <= 3 stored as the nibble v reads as v / 2 in E2M1, and
    the weight codes -4..4 all have exact E2M1 encodings."""
    v = np.arange(4)
    assert np.array_equal(_e2m1_value(v), v / 2.0)
    vals = _e2m1_value(np.arange(16))
    for w in range(-4, 5):
        assert w in vals
    # the block scale 2^-4 on both operands turns (v/2) * w into v * w * 2^-9
    assert (0.5 * 2.0 ** -4) * 2.0 ** -4 == 2.0 ** -9


@pytest.mark.parametrize("shape", [(2, 64, 3, 64, 2), (4, 96, 1, 128, 3), (1, 288, 3, 64, 2), (2, 32, 3, 192, 3)])
def test_fp4_pack_unpack_roundtrip_and_e2m1_encoding(shape):
    G, Co, k, Ci, bits_w = shape
    d = B.layer_desc(1, 8, 8, G, Ci, Co, k, 1, k // 2, 2, bits_w, 2, code_format=B.PQ_CODES_C32F4)
    gen = synth.generator(sum(shape) + 5)
    wq = synth.random_codes((G, Co, k, k, Ci), bits_w, gen, signed=True)
    packed = B.palquant_pack_weight_codes_host(wq, d)
    assert packed.size == wq.size // 2
    assert np.array_equal(B.palquant_unpack_weight_codes_host(packed, d), wq)
    nibbles = np.stack([packed & 15, packed >> 4], axis=-1).ravel()
    assert np.array_equal(np.sort(_e2m1_value(nibbles)), np.sort(wq.ravel().astype(np.float64)))


def test_fp4_layout_rules():
    F4 = B.PQ_CODES_C32F4
    ok = B.palquant_conv_plan(B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 3, 2, code_format=F4))
    assert ok.supported == 1 and ok.k_chunk % 64 == 0
    for d in [B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 3, 2, 2, code_format=F4),   # 3-bit activations
              B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 4, 2, code_format=F4),   # 4-bit weights
              B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 2, 3, code_format=F4),   # 3-bit output codes
              B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=F4),   # Cin_g % 64 != 0
              B.layer_desc(1, 8, 8, 2, 64, 48, 3, 1, 1, 2, 2, 2, code_format=F4)]:  # Cout_g % 32 != 0
        assert B.palquant_conv_plan(d).supported == 0
    d = B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 2, 2, code_format=F4)
    with pytest.raises(B.PalquantError) as e:   # a per-channel scatter cannot write nibbles
        B.palquant_layer_fused(16, 16, d, [1.0] * 2, [1.0] * 2, shuf=B.shuffle(2, 0), q_out_dev=16)
    assert e.value.status == B.PQ_EUNSUPPORTED
    with pytest.raises(B.PalquantError) as e:   # bit-decomposed slices are one per byte
        B.palquant_bitsplit_desc(d, 1)
    assert e.value.status == B.PQ_EUNSUPPORTED
    w = np.zeros((2, 32, 3, 3, 64), np.float32)
    with pytest.raises(B.PalquantError) as e:   # odd levels +-5, +-7 are not E2M1 values
        B.palquant_pack_weights_odd_host(w, B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 3, 2, code_format=F4),
                                         [1.0, 1.0])
    assert e.value.status == B.PQ_EUNSUPPORTED
    with pytest.raises(B.PalquantError) as e:   # the quantiser's FP4 output holds 2-bit codes
        B.palquant_quantize_act(16, 16, 1, 4, 4, 2, 32, 3, [1.0, 1.0], code_format=F4)
    assert e.value.status == B.PQ_EINVAL


F4_LAYERS = [c for c in ALL_LAYERS if c.bits_a <= 2 and c.bits_out <= 2 and c.bits_w <= 3 and c.Cin_g % 64 == 0
             and c.Cout_g % 32 == 0]


@pytest.mark.parametrize("c", F4_LAYERS, ids=lambda c: f"{c.H}x{c.W}k{c.k}s{c.stride}G{c.G}c{c.Cin_g}-{c.Cout_g}")
def test_fp4_plan_invariants(c):
    plan = B.palquant_conv_plan(_desc(c, code_format=B.PQ_CODES_C32F4))
    assert plan.supported == 1
    assert plan.smem_bytes + 1024 <= 227 * 1024
    assert plan.n_block * plan.n_blocks == c.Cout_g and plan.n_block % 16 == 0 and plan.n_block <= 128
    assert plan.k_chunk * plan.k_blocks == c.Cin_g and plan.k_chunk % 64 == 0
    # accumulators and the 32 scale-factor columns share the 512 TMEM columns
    npow2 = 1 << (plan.n_block - 1).bit_length()
    assert plan.acc_stages * plan.m_tiles * npow2 + 32 <= 512


def test_fp4_code_helpers_roundtrip():
    from layer_cases import c32f4_to_nhwc, code_bytes, from_format, to_format

    gen = synth.generator(78)
    q = synth.random_codes((2, 3, 4, 64), 2, gen)
    raw = to_format(q, 4)
    assert raw.size == code_bytes(q.size, 4) == q.size // 2
    assert np.array_equal(c32f4_to_nhwc(raw, 2, 3, 4, 64), q)
    assert np.array_equal(from_format(raw, 4, 2, 3, 4, 64), q)
    # channel c of a position: byte (c % 32) / 2 of its block's 16-byte row, low
    # nibble for even c; the second 32-channel block lies H*W*16 bytes further on
    one = np.zeros((1, 2, 1, 64), np.uint8)
    one[0, 1, 0, 32 + 7] = 3
    r = to_format(one, 4)
    assert np.flatnonzero(r).tolist() == [2 * 16 + 16 + 3] and r[2 * 16 + 16 + 3] == 3 << 4


def test_quantize_layer_fused_rules():
    """Quantise-on-load covers stride-1 layers with byte or FP4 codes out; the
    reciprocal steps are required and must be finite and non-negative."""
    d = B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=B.PQ_CODES_C16)
    for bad in [B.layer_desc(1, 8, 8, 2, 32, 32, 3, 2, 1, 2, 2, 2, code_format=B.PQ_CODES_C16),    # stride 2
                B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=B.PQ_CODES_C16P2),  # packed codes
                B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1, 2, 2, 2, code_format=B.PQ_CODES_C32F4)]:  # FP4, Cin_g 32
        with pytest.raises(B.PalquantError) as e:
            B.palquant_quantize_layer_fused(16, [1.0, 1.0], 16, bad, [1.0] * 2, [1.0] * 2, q_out_dev=16)
        assert e.value.status == B.PQ_EUNSUPPORTED
    with pytest.raises(B.PalquantError) as e:
        B.palquant_quantize_layer_fused(16, [1.0, float("nan")], 16, d, [1.0] * 2, [1.0] * 2, q_out_dev=16)
    assert e.value.status == B.PQ_EINVAL
    with pytest.raises(B.PalquantError) as e:
        B.palquant_quantize_layer_fused(16, [1.0, -2.0], 16, d, [1.0] * 2, [1.0] * 2, q_out_dev=16)
    assert e.value.status == B.PQ_EINVAL
    # one packing serves both the plain layer and quantise-on-load (tap-major layout)
    gen = synth.generator(9)
    wq = synth.random_codes((2, 32, 3, 3, 64), 2, gen, signed=True)
    d2 = B.layer_desc(1, 8, 8, 2, 64, 32, 3, 1, 1, 2, 2, 2, code_format=B.PQ_CODES_C16)
    assert np.array_equal(B.palquant_unpack_weight_codes_host(B.palquant_pack_weight_codes_host(wq, d2), d2), wq)


# ------------------------------------------------ quantisation-aware training (host checks)
def test_fake_quant_argument_rules():
    """Invalid arguments return before any launch (no device memory is touched)."""
    A = 0x10000  # a 16-byte aligned stand-in address: every case below fails its checks first
    ok = dict(P=8, G=2, Cg=8, bits=2, kind=0, l=[0.0, 0.0], u=[1.0, 2.0])

    def fwd(**kw):
        a = dict(ok, **kw)
        return B.lib.palquant_fake_quant_forward(A, A, a["P"], a["G"], a["Cg"], a["bits"], a["kind"],
                                                 B._ptr(B._f32(a["l"])), B._ptr(B._f32(a["u"])), None)

    bad = [dict(Cg=6), dict(Cg=0), dict(G=0), dict(G=65, l=[0.0] * 65, u=[1.0] * 65), dict(bits=0), dict(bits=9),
           dict(kind=2), dict(P=-1), dict(l=[0.0, 2.0]), dict(l=[0.0, float("nan")]), dict(u=[1.0, float("inf")]),
           dict(l=[1.0, 0.0], u=[1.0, 2.0])]
    for kw in bad:
        assert fwd(**kw) == B.PQ_EINVAL, kw
    assert B.lib.palquant_fake_quant_forward(A + 4, A, 8, 2, 8, 2, 0, B._ptr(B._f32(ok["l"])),
                                             B._ptr(B._f32(ok["u"])), None) == B.PQ_EINVAL
    # more than 2^32 float4s per group
    assert fwd(P=1 << 31, Cg=16) == B.PQ_EUNSUPPORTED
    assert B.palquant_fake_quant_scratch_bytes(1 << 31, 1, 16) == 0
    # backward: a scratch buffer too small, misaligned gradient outputs
    sb = B.palquant_fake_quant_scratch_bytes(8, 2, 8)
    assert sb >= 2 * 16
    lp, up = B._ptr(B._f32(ok["l"])), B._ptr(B._f32(ok["u"]))
    assert B.lib.palquant_fake_quant_backward(A, A, A, A, A, 8, 2, 8, 2, 0, lp, up, A, sb - 1, None) == B.PQ_EINVAL
    assert B.lib.palquant_fake_quant_backward(A, A, A, A + 4, A, 8, 2, 8, 2, 0, lp, up, A, sb, None) == B.PQ_EINVAL
    assert B.lib.palquant_fake_quant_backward(A, A, A, A, A, 8, 2, 6, 2, 0, lp, up, A, sb, None) == B.PQ_EINVAL
