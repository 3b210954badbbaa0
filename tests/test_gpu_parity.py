"""GPU parity of the hot path against the CPU oracle, through the C ABI.

Integer outputs (activation codes, int32 sums, requantised codes) must match the
oracle bit for bit; fp32 outputs within a relative error of 1e-5 (they are single
IEEE multiplies / adds in the same order, so they are expected to be exact).
"""
import numpy as np
import pytest

import oracle
from paper_2208_01944_gb300 import synth, workloads

from layer_cases import Case, assert_layer_parity, prepare, run_gpu

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2208_01944_gb300 import binding

    return binding


# ------------------------------------------------------------ a2 quantize
@pytest.mark.parametrize("shape,G,bits", [((2, 7, 9, 64), 4, 2), ((1, 5, 5, 3 * 16), 3, 4), ((3, 4, 6, 2 * 20), 2, 3),
                                          ((1, 1, 1, 32), 1, 8), ((5, 33, 17, 256), 4, 2)])
def test_quantize_act_matches_oracle(B, shape, G, bits):
    gen = synth.generator(sum(shape) + bits)
    x = synth.normal(shape, gen, 2.0)
    flat = x.reshape(-1)
    # ties, NaN and infinities at fixed places
    specials = np.array([0.5, 1.5, 2.5, -0.5, np.nan, np.inf, -np.inf, 3.5, 1e30, -0.0], dtype=np.float32)
    flat[: specials.size] = specials
    inv = (synth.half_normal((G,), gen) + 0.5).astype(np.float32)
    inv[0] = 1.0
    ref = oracle.quantize_act(x, G, bits, inv)
    xd = torch.from_numpy(x).cuda()
    q = torch.full(shape, 254, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(xd, q, shape[0], shape[1], shape[2], G, shape[3] // G, bits, inv)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(q.cpu().numpy(), ref)


def test_quantize_act_misaligned_views_use_scalar_path(B):
    gen = synth.generator(3)
    x = synth.normal((1, 4, 4, 33), gen)
    xd = torch.from_numpy(x).cuda()
    # an offset view: 4-byte aligned but not 16-byte aligned
    big = torch.zeros(x.size + 1, dtype=torch.float32, device="cuda")
    big[1:] = xd.reshape(-1)
    q = torch.zeros(x.size + 1, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(big[1:].data_ptr(), q[1:].data_ptr(), 1, 4, 4, 1, 33, 2, [1.7])
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(q[1:].cpu().numpy().reshape(x.shape), oracle.quantize_act(x, 1, 2, [1.7]))


# ------------------------------------------------------------ a0 steps
@pytest.mark.parametrize("shape,G,bits", [((2, 9, 7, 64), 2, 2), ((64, 8, 8, 256), 4, 2), ((1, 3, 3, 24), 3, 4)])
def test_act_steps_match_oracle(B, shape, G, bits):
    gen = synth.generator(11)
    x = synth.half_normal(shape, gen)
    xd = torch.from_numpy(x).cuda()
    P = shape[0] * shape[1] * shape[2]
    nbytes = B.palquant_act_steps_scratch_bytes(P, G)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    s = B.palquant_act_steps(xd, shape[0], shape[1], shape[2], G, shape[3] // G, bits, scratch, nbytes)
    ref = oracle.act_step(x, G, bits)
    # both sum in double (different order), then round to float once: at most 1 ulp apart
    assert np.all(np.abs(s.view(np.int32) - ref.view(np.int32)) <= 1)


# ------------------------------------------------------------ a3-a6 layer
SMALL_CASES = [
    Case(1, 28, 28, 2, 32, 32, 3, 1, 1, seed=0),                      # config 0 shape
    Case(2, 13, 11, 3, 32, 48, 3, 1, 1, seed=1),                      # odd sizes, 3 output chunks
    Case(3, 9, 17, 4, 64, 64, 3, 2, 1, seed=2),                       # stride 2, odd input
    Case(2, 10, 10, 2, 64, 128, 1, 2, 0, kind=0, relu=False, seed=3),  # 1x1 stride-2 downsample
    Case(2, 7, 9, 4, 96, 96, 1, 1, 0, seed=4),                        # flat mode, ragged last tile
    Case(1, 15, 15, 1, 32, 16, 3, 1, 0, bits=4, kind=0, seed=5),      # pad 0, G = 1, 4-bit
    Case(2, 14, 14, 8, 32, 32, 3, 1, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=6),
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, bits=4, seed=7),            # streamed weights, 4-bit
    Case(1, 7, 7, 2, 512, 32, 3, 1, 1, seed=8),                       # four K blocks, whole-image tiles
    Case(2, 8, 8, 2, 32, 320, 3, 1, 1, seed=9),                       # two output-channel blocks
    Case(1, 5, 130, 1, 32, 16, 3, 1, 1, seed=10),                     # row wider than 128 positions
    Case(2, 9, 9, 4, 32, 32, 3, 1, 1, kind=2, seed=11),               # channel shuffle
    Case(2, 11, 10, 2, 64, 64, 3, 1, 1, shortcut=True, seed=12),      # shortcut add before ReLU
    Case(1, 9, 11, 2, 32, 64, 5, 1, 2, seed=13),                      # 5x5 kernel
    Case(2, 6, 6, 2, 32, 32, 3, 1, 1, bits=3, bits_out=4, relu=False, kind=1, shift=-1, seed=14),
    Case(1, 16, 16, 4, 64, 64, 3, 2, 0, seed=15),                     # stride 2 without padding
    Case(2, 36, 40, 2, 64, 64, 3, 1, 1, shortcut=True, seed=16),      # three accumulators per tile (c16)
    Case(1, 30, 20, 2, 64, 64, 3, 1, 1, seed=17),                     # three accumulators, ragged last tile
    Case(1, 40, 30, 2, 64, 64, 3, 2, 1, seed=18),                     # three accumulators, stride 2
    Case(2, 20, 20, 2, 64, 64, 1, 1, 0, seed=19),                     # flat, two boxes per tile, ragged
    Case(2, 17, 17, 2, 64, 64, 1, 1, 0, shortcut=True, seed=20),      # flat, second box wholly past the image
    Case(1, 6, 140, 2, 32, 32, 3, 2, 1, seed=21),                     # stride 2, window wider than one TMA box row
    Case(2, 11, 10, 2, 32, 48, 3, 1, 1, shortcut=True, seed=22),      # shortcut with int32 sums, 16-column units
    Case(2, 13, 15, 2, 32, 32, 5, 2, 2, seed=23),                     # 5x5 stride 2: a window of 4 phases, 3 taps each way
]


FORMATS = [0, 2]  # NHWC codes, channel-blocked codes


@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("c", SMALL_CASES, ids=str)
def test_layer_fused_matches_oracle(B, c, fmt):
    ref = prepare(c)
    got = run_gpu(c, ref, fmt=fmt)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("shape,G,bits", [((2, 7, 9, 64), 4, 2), ((3, 5, 6, 3 * 16), 3, 4), ((1, 1, 1, 32), 1, 8),
                                         # several 256-channel ranges and ragged pixel tiles; a ragged range
                                         ((2, 11, 13, 768), 4, 2), ((1, 40, 40, 400), 5, 3)])
def test_quantize_act_c16_matches_oracle(B, shape, G, bits):
    from layer_cases import c16_to_nhwc

    gen = synth.generator(sum(shape) + 7)
    x = synth.normal(shape, gen, 2.0)
    x.reshape(-1)[:6] = np.array([0.5, 1.5, 2.5, np.nan, np.inf, -np.inf], dtype=np.float32)
    inv = (synth.half_normal((G,), gen) + 0.5).astype(np.float32)
    xd = torch.from_numpy(x).cuda()
    q = torch.full(shape, 254, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(xd, q, shape[0], shape[1], shape[2], G, shape[3] // G, bits, inv, code_format=B.PQ_CODES_C16)
    assert B.palquant_sync_check() == B.PQ_OK
    got = c16_to_nhwc(q.cpu().numpy(), *shape)
    assert np.array_equal(got, oracle.quantize_act(x, G, bits, inv))


def test_group_conv_matches_oracle(B):
    c = Case(2, 12, 9, 3, 64, 48, 3, 1, 1, kind=0)
    ref = prepare(c)
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad)
    q = torch.from_numpy(ref["q"]).cuda()
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(ref["wq"], d)).cuda()
    acc = torch.zeros((c.N, c.Ho, c.Wo, c.G * c.Cout), dtype=torch.int32, device="cuda")
    B.palquant_group_conv(q, wp, acc, d)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), oracle.group_conv(ref["q"], ref["wq"], c.stride, c.pad))


@pytest.mark.parametrize("bits,Cin", [(4, 512), (2, 512), (4, 64)])
def test_worst_case_magnitudes_exact(B, bits, Cin):
    """All codes at their extreme: every sum is the largest the layer can produce."""
    G, Co, k = 2, 32, 3
    N, H, W = 1, 6, 6
    qa, wmin = (1 << bits) - 1, -(1 << (bits - 1))
    q = np.full((N, H, W, G * Cin), qa, dtype=np.uint8)
    wq = np.full((G, Co, k, k, Cin), wmin, dtype=np.int8)
    wq[1] = (1 << (bits - 1)) - 1
    d = B.layer_desc(N, H, W, G, Cin, Co, k, 1, 1, bits, bits, bits)
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).cuda()
    acc = torch.zeros((N, H, W, G * Co), dtype=torch.int32, device="cuda")
    B.palquant_group_conv(torch.from_numpy(q).cuda(), wp, acc, d)
    assert B.palquant_sync_check() == B.PQ_OK
    ref = oracle.group_conv(q, wq, 1, 1)
    assert np.abs(ref).max() == 9 * Cin * qa * -wmin
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)


def test_empty_batch_is_a_noop(B):
    d = B.layer_desc(0, 8, 8, 2, 32, 32, 3, 1, 1)
    wq = np.zeros((2, 32, 3, 3, 32), dtype=np.int8)
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).cuda()
    q = torch.zeros(16, dtype=torch.uint8, device="cuda")
    acc = torch.zeros(16, dtype=torch.int32, device="cuda")
    B.palquant_group_conv(q, wp, acc, d)
    assert B.palquant_sync_check() == B.PQ_OK


def test_outputs_untouched_outside_tensor(B):
    """Canary bytes around the outputs stay intact (no out-of-bounds stores)."""
    c = Case(2, 9, 13, 2, 32, 48, 3, 1, 1, seed=21)
    ref = prepare(c)
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad)
    n_out = c.N * c.Ho * c.Wo * c.G * c.Cout
    pad = 4096
    q = torch.from_numpy(ref["q"]).cuda()
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(ref["wq"], d)).cuda()
    qo = torch.full((n_out + 2 * pad,), 0xA5, dtype=torch.uint8, device="cuda")
    y = torch.full((n_out + 2 * pad // 4 * 4,), 7.25, dtype=torch.float32, device="cuda")
    B.palquant_layer_fused(q, wp, d, ref["m_out"], ref["m_req"], B.shuffle(1, 1), None, None,
                           y[pad // 4 * 2: pad // 4 * 2 + n_out].data_ptr(), qo[pad: pad + n_out].data_ptr())
    assert B.palquant_sync_check() == B.PQ_OK
    qh = qo.cpu().numpy()
    assert (qh[:pad] == 0xA5).all() and (qh[pad + n_out:] == 0xA5).all()
    yh = y.cpu().numpy()
    assert (yh[: pad // 2] == 7.25).all() and (yh[pad // 2 + n_out:] == 7.25).all()
    assert np.array_equal(qh[pad: pad + n_out].reshape(-1, c.G * c.Cout), ref["q_ref"])


# ----------------------------------------------- full-size workloads (sampled)
def _sample_pixels(N, Ho, Wo, n_random, seed):
    rng = np.random.default_rng(seed)
    P = N * Ho * Wo
    corners = []
    for n in (0, N - 1):
        for oh in (0, Ho - 1):
            for ow in (0, Wo - 1):
                corners.append((n * Ho + oh) * Wo + ow)
    edges = [(n * Ho + oh) * Wo + ow for n in (N // 2,) for oh in range(Ho) for ow in (0, Wo - 1)]
    pix = np.unique(np.concatenate([np.array(corners + edges), rng.integers(0, P, n_random)]))
    return pix.astype(np.int64)


FULL = [("config1", workloads.CONFIG1)] + [(f"config3_{i}", c) for i, c in enumerate(workloads.CONFIG3)] + [
    ("config4", workloads.CONFIG4)]


@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("name,cfg", FULL, ids=[n for n, _ in FULL])
def test_full_size_layer_sampled(B, name, cfg, fmt):
    c = Case(cfg.N, cfg.H, cfg.W, cfg.G, cfg.Cin_g, cfg.Cout_g, cfg.k, cfg.stride, cfg.pad, bits=cfg.bits_a,
             kind=cfg.shuffle_kind, shift=cfg.shuffle_shift, relu=cfg.relu, seed=0)
    pix = _sample_pixels(c.N, c.Ho, c.Wo, 3000, 1)
    ref = prepare(c, sample_pix=pix)
    got = run_gpu(c, ref, fmt=fmt)
    assert_layer_parity(c, ref, got, pix)


@pytest.mark.parametrize("name,cfg", FULL, ids=[n for n, _ in FULL])
def test_full_size_codes_only_c16_sampled(B, name, cfg):
    """The benchmarked configuration: channel-blocked codes in and out, codes only."""
    c = Case(cfg.N, cfg.H, cfg.W, cfg.G, cfg.Cin_g, cfg.Cout_g, cfg.k, cfg.stride, cfg.pad, bits=cfg.bits_a,
             kind=cfg.shuffle_kind, shift=cfg.shuffle_shift, relu=cfg.relu, seed=0)
    pix = _sample_pixels(c.N, c.Ho, c.Wo, 3000, 2)
    ref = prepare(c, sample_pix=pix)
    got = run_gpu(c, ref, outputs=("q",), fmt=2)
    assert_layer_parity(c, ref, got, pix)


# ------------------------------- the pointwise kernel (1x1 layers, codes only out)
PW_CASES = [
    Case(2, 7, 7, 4, 32, 16, 1, seed=150),                            # 49 pixels: one accumulator, ragged
    Case(3, 14, 14, 4, 96, 96, 1, seed=151),                          # the config-4 shape: 196 of 256 rows
    Case(2, 20, 20, 2, 64, 64, 1, seed=152),                          # 400 pixels: tiles of 256 and 144
    Case(1, 16, 16, 1, 32, 256, 1, kind=0, seed=153),                 # N = 256: tiles of 128 pixels
    Case(2, 9, 13, 8, 32, 48, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=154),  # odd plane count
    Case(2, 12, 12, 2, 64, 32, 1, bits=4, bits_out=3, relu=False, shift=-1, seed=155),
    Case(1, 1, 1, 2, 32, 16, 1, seed=156),                            # one pixel
    Case(4, 8, 8, 1, 256, 64, 1, kind=0, seed=157),                   # eight K steps
    Case(1, 30, 30, 3, 32, 32, 1, seed=158),                          # 900 pixels, three groups
    Case(5, 11, 23, 2, 128, 16, 1, bits_out=1, seed=159),             # N = 16: four accumulator stages, 1-bit codes out
]


@pytest.mark.parametrize("c", PW_CASES, ids=str)
def test_pointwise_kernel_matches_oracle(B, c):
    """1x1 layers with channel-blocked codes in and codes only out run on the
    pointwise kernel; its codes equal the oracle's bit for bit."""
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, 1, 1, 0, c.bits, c.bits, c.bo, int(c.relu),
                     code_format=B.PQ_CODES_C16)
    assert B.palquant_conv_plan(d).pointwise == 1
    ref = prepare(c)
    assert_layer_parity(c, ref, run_gpu(c, ref, outputs=("q",), fmt=2))


def test_pointwise_not_taken_when_weights_do_not_fit(B):
    """Weights beyond the pointwise kernel's resident budget (96 KB) go to the
    general kernel, with the same results."""
    c = Case(1, 9, 9, 4, 128, 256, 1, seed=160)                      # 4 x 128 x 256 = 128 KB of weights
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, 1, 1, 0, c.bits, c.bits, c.bo, int(c.relu),
                     code_format=B.PQ_CODES_C16)
    assert B.palquant_conv_plan(d).pointwise == 0
    ref = prepare(c)
    assert_layer_parity(c, ref, run_gpu(c, ref, outputs=("q",), fmt=2))


def test_pointwise_inputs_ready_chain(B):
    """PQ_LAYER_INPUTS_READY over a chain of pointwise layers L1 -> L2 -> L3: L2
    reads nothing L1 writes, L3 reads L1's codes.  L1 fills every SM, L2 is a few
    CTAs.  L3's codes equal the oracle's layer over the oracle's L1 codes, and
    back-to-back flagged launches over independent inputs equal flagless ones."""
    from layer_cases import from_format, to_format

    fmt = B.PQ_CODES_C16
    G = 4
    c1 = Case(64, 14, 14, G, 96, 96, 1, seed=161)
    c2 = Case(1, 4, 4, G, 96, 96, 1, seed=162)
    r1, r2 = prepare(c1), prepare(c2)
    gen = synth.generator(163)
    w3 = synth.he_weights(G, 32, 1, 1, c1.Cout, gen)
    s_w3 = oracle.weight_step(w3, 2)
    inv_sw3 = oracle.inv_step(s_w3)
    s_a3 = np.full(G, 0.75, np.float32)
    m_out3, m_req3 = oracle.epilogue_scales(s_w3, s_a3, s_a3, 1.0, 1, 1)
    q1_ref = r1["q_ref"].reshape(c1.N, c1.H, c1.W, G * c1.Cout)
    acc3 = oracle.group_conv(q1_ref, oracle.quantize_weights(w3, 2, inv_sw3), 1, 0).reshape(-1, G * 32)
    _, _, q3_ref = oracle.epilogue(acc3, G, m_out3, m_req3, 1, 1, None, None, True, 2)

    def desc(c, cin, cout, flags):
        return B.layer_desc(c.N, c.H, c.W, G, cin, cout, 1, 1, 0, 2, 2, 2, 1, code_format=fmt, flags=flags)

    d1 = desc(c1, 96, 96, 0)
    d2 = desc(c2, 96, 96, B.PQ_LAYER_INPUTS_READY)
    d3 = desc(c1, 96, 32, B.PQ_LAYER_INPUTS_READY)
    assert all(B.palquant_conv_plan(d).pointwise == 1 for d in (d1, d2, d3))
    wps = []
    for d, w, inv in ((d1, r1["w"], r1["inv_sw"]), (d2, r2["w"], r2["inv_sw"]), (d3, w3, inv_sw3)):
        nb = B.palquant_packed_weight_bytes(d)
        wp = torch.empty(nb, dtype=torch.uint8, device="cuda")
        B.palquant_pack_weights(w, d, inv, wp, nb)
        wps.append(wp)
    q1 = torch.from_numpy(to_format(r1["q"], fmt)).cuda()
    q2 = torch.from_numpy(to_format(r2["q"], fmt)).cuda()
    shuf = B.shuffle(1, 1)
    o2 = torch.empty(c2.N * c2.H * c2.W * G * 96, dtype=torch.uint8, device="cuda")
    for rep in range(3):
        o1 = torch.full((c1.N * c1.H * c1.W * G * 96,), 255, dtype=torch.uint8, device="cuda")
        o3 = torch.full((c1.N * c1.H * c1.W * G * 32,), 255, dtype=torch.uint8, device="cuda")
        B.palquant_layer_fused(q1, wps[0], d1, r1["m_out"], r1["m_req"], shuf, None, None, None, o1)
        B.palquant_layer_fused(q2, wps[1], d2, r2["m_out"], r2["m_req"], shuf, None, None, None, o2)
        B.palquant_layer_fused(o1, wps[2], d3, m_out3, m_req3, shuf, None, None, None, o3)
        assert B.palquant_sync_check() == B.PQ_OK
        assert np.array_equal(from_format(o1.cpu().numpy(), fmt, c1.N, c1.H, c1.W, G * 96), q1_ref), rep
        got3 = from_format(o3.cpu().numpy(), fmt, c1.N, c1.H, c1.W, G * 32).reshape(-1, G * 32)
        assert np.array_equal(got3, q3_ref), rep
    # back to back over independent inputs (five launches, two output buffers in turn)
    d1r = desc(c1, 96, 96, B.PQ_LAYER_INPUTS_READY)
    outs = [torch.full((c1.N * c1.H * c1.W * G * 96,), 255, dtype=torch.uint8, device="cuda") for _ in range(2)]
    qs = [q1, torch.flip(q1, dims=[0]).contiguous()]
    for i in range(5):
        B.palquant_layer_fused(qs[i % 2], wps[0], d1r, r1["m_out"], r1["m_req"], shuf, None, None, None, outs[i % 2])
    assert B.palquant_sync_check() == B.PQ_OK
    for i in (3, 4):
        single = torch.full_like(outs[0], 255)
        B.palquant_layer_fused(qs[i % 2], wps[0], d1, r1["m_out"], r1["m_req"], shuf, None, None, None, single)
        assert B.palquant_sync_check() == B.PQ_OK
        assert torch.equal(outs[i % 2], single), i


# ------------------------------------------------------ failure detection
def test_watchdog_times_out_and_context_survives(B):
    assert B.palquant_watchdog_selftest(2_000_000) == B.PQ_ETIMEOUT  # a 2 ms wait nobody completes
    assert B.palquant_sync_check() == B.PQ_OK                         # the error word was cleared
    c = Case(1, 6, 6, 2, 32, 32, 3, 1, 1, seed=30)
    ref = prepare(c)
    assert_layer_parity(c, ref, run_gpu(c, ref))                      # the context still works


# ------------------------------------------- codes-only path (the timed one)
CODES_ONLY = [
    Case(2, 13, 11, 3, 32, 48, 3, 1, 1, seed=40),
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, bits=4, seed=41),
    Case(2, 7, 9, 4, 96, 96, 1, 1, 0, seed=42),
    Case(3, 9, 17, 4, 64, 64, 3, 2, 1, seed=43),
    Case(2, 17, 17, 4, 96, 96, 1, 1, 0, seed=45),                     # flat, two boxes per tile
]


# Shortcut layers writing fp32 and codes but no int32 sums: the epilogue fetches the
# next unit's shortcut rows while the current unit computes (two staging buffers a
# warp).  16-column units (48 and 80 output channels), several units per warpgroup,
# rows outside the output, stride 2, the channel shuffle and the cyclic shuffle.
SHORTCUT_YQ = [
    Case(2, 13, 11, 2, 32, 48, 3, 1, 1, shortcut=True, seed=50),
    Case(1, 9, 10, 2, 64, 80, 3, 1, 1, shortcut=True, kind=1, shift=-1, seed=51),
    Case(2, 36, 40, 2, 64, 64, 3, 1, 1, shortcut=True, seed=52),
    Case(2, 12, 14, 2, 64, 128, 3, 2, 1, shortcut=True, seed=53),
    Case(2, 9, 9, 4, 32, 32, 3, 1, 1, shortcut=True, kind=2, seed=54),
    Case(2, 7, 9, 2, 96, 96, 1, 1, 0, shortcut=True, relu=False, seed=55),
]


@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("c", SHORTCUT_YQ, ids=str)
def test_layer_shortcut_y_and_codes_matches_oracle(B, c, fmt):
    ref = prepare(c)
    got = run_gpu(c, ref, outputs=("y", "q"), fmt=fmt)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("c", CODES_ONLY, ids=str)
def test_layer_codes_only_matches_oracle(B, c, fmt):
    ref = prepare(c)
    got = run_gpu(c, ref, outputs=("q",), fmt=fmt)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("k", [3, 1], ids=["3x3", "1x1"])
@pytest.mark.parametrize("fmt,bits", [(0, 4), (2, 4), (2, 1), (4, 2)], ids=["nhwc4", "c16_4", "c16_1", "fp4_2"])
@pytest.mark.parametrize("mult", [0.5, 0.25, 1.0 / 3.0, 1e4, -0.5, 1e-3])
def test_requant_ties_round_half_even(B, mult, fmt, bits, k):
    """Multipliers that put many products exactly on .5 (ties must round to even),
    that saturate every positive sum, that make every product negative, and that
    round almost everything to 0; codes only, in every code format (1x1 layers
    with channel-blocked byte codes run on the pointwise kernel)."""
    c = Case(2, 10, 10, 2, 64, 64, k, 1, (k - 1) // 2, bits=bits if bits > 1 else 2, bits_out=bits, seed=44)
    ref = prepare(c)
    m_req = np.array([mult, mult * 0.75], dtype=np.float32)
    acc = oracle.group_conv(ref["q"], ref["wq"], c.stride, c.pad).reshape(-1, c.G * c.Cout)
    _, _, q_ref = oracle.epilogue(acc, c.G, ref["m_out"], m_req, c.kind, c.shift, None, None, True, bits)
    ref = dict(ref, m_req=m_req, q_ref=q_ref)
    got = run_gpu(c, ref, outputs=("q",), fmt=fmt)
    assert np.array_equal(got["q_out"], q_ref)
    if mult == 0.5:
        assert np.any((acc % 2 == 1) & (acc > 0)), "the case must contain ties"
    if mult == 1e4:
        assert np.any(q_ref == (1 << bits) - 1) and np.any(acc > 0)


# ------------------------------------ packed 2-bit channel-blocked codes (format 3)
P2_CASES = [
    Case(1, 28, 28, 2, 32, 32, 3, 1, 1, seed=50),
    Case(2, 12, 16, 3, 32, 48, 3, 1, 1, seed=51),                     # 3 output chunks
    Case(2, 8, 8, 4, 96, 96, 1, 1, 0, seed=52),                       # flat, one partial tile
    Case(2, 14, 14, 4, 96, 96, 1, 1, 0, seed=53),                     # flat, ragged second tile
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, seed=54),                   # streamed weights
    Case(1, 8, 8, 2, 512, 32, 3, 1, 1, seed=55),                      # four K blocks
    Case(2, 8, 8, 2, 32, 320, 3, 1, 1, seed=56),                      # two output-channel blocks
    Case(1, 5, 132, 1, 32, 16, 3, 1, 1, seed=57),                     # rows wider than 128 positions
    Case(2, 12, 8, 2, 64, 64, 3, 1, 1, shortcut=True, seed=58),       # shortcut add
    Case(1, 9, 12, 2, 32, 64, 5, 1, 2, seed=59),                      # 5x5, pad 2 (staging offset 2)
    Case(1, 16, 16, 1, 32, 16, 3, 1, 0, kind=0, seed=60),             # pad 0 (offset 0)
    Case(2, 8, 12, 8, 32, 32, 3, 1, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=61),
    Case(2, 6, 8, 2, 32, 32, 3, 1, 1, relu=False, kind=1, shift=-1, seed=62),
]


@pytest.mark.parametrize("c", P2_CASES, ids=str)
def test_layer_fused_packed_codes_matches_oracle(B, c):
    ref = prepare(c)
    got = run_gpu(c, ref, fmt=B.PQ_CODES_C16P2)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("c", P2_CASES[:6], ids=str)
def test_layer_codes_only_packed_matches_oracle(B, c):
    ref = prepare(c)
    got = run_gpu(c, ref, outputs=("q",), fmt=B.PQ_CODES_C16P2)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("name,cfg", [(n, c) for n, c in FULL if c.bits_a <= 2], ids=lambda v: v if isinstance(v, str) else "")
def test_full_size_codes_only_packed_sampled(B, name, cfg):
    c = Case(cfg.N, cfg.H, cfg.W, cfg.G, cfg.Cin_g, cfg.Cout_g, cfg.k, cfg.stride, cfg.pad, bits=cfg.bits_a,
             kind=cfg.shuffle_kind, shift=cfg.shuffle_shift, relu=cfg.relu, seed=0)
    pix = _sample_pixels(c.N, c.Ho, c.Wo, 3000, 3)
    ref = prepare(c, sample_pix=pix)
    got = run_gpu(c, ref, outputs=("q",), fmt=B.PQ_CODES_C16P2)
    assert_layer_parity(c, ref, got, pix)


@pytest.mark.parametrize("shape,G,bits", [((2, 7, 9, 64), 4, 2), ((1, 5, 6, 48), 3, 1), ((2, 11, 13, 768), 4, 2)])
def test_quantize_act_packed_matches_oracle(B, shape, G, bits):
    from layer_cases import c16p2_to_nhwc

    gen = synth.generator(sum(shape) + 9)
    x = synth.normal(shape, gen, 2.0)
    x.reshape(-1)[:6] = np.array([0.5, 1.5, 2.5, np.nan, np.inf, -np.inf], dtype=np.float32)
    inv = (synth.half_normal((G,), gen) + 0.5).astype(np.float32)
    q = torch.full((int(np.prod(shape)) // 4,), 254, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(torch.from_numpy(x).cuda(), q, shape[0], shape[1], shape[2], G, shape[3] // G, bits, inv,
                            code_format=B.PQ_CODES_C16P2)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(c16p2_to_nhwc(q.cpu().numpy(), *shape), oracle.quantize_act(x, G, bits, inv))


# ---------------------------------------- the paper's odd weight levels (Eq. 2-3)
@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("bits_w", [2, 3])
def test_layer_with_odd_weight_levels_matches_oracle(B, fmt, bits_w):
    from layer_cases import from_format

    N, H, W, G, Ci, Co = 2, 12, 10, 2, 64, 48
    gen = synth.generator(70 + bits_w)
    x = synth.half_normal((N, H, W, G * Ci), gen)
    w = synth.he_weights(G, Co, 3, 3, Ci, gen)
    s_a = oracle.act_step(x, G, 2)
    inv_s = oracle.inv_step(s_a)
    u = (2.0 * np.abs(w).reshape(G, -1).mean(axis=1)).astype(np.float32)
    s_w = (u.astype(np.float64) / ((1 << bits_w) - 1)).astype(np.float32)  # de-quantised weight = code * s_w
    q = oracle.quantize_act(x, G, 2, inv_s)
    wq = oracle.quantize_weights_odd(w, bits_w, u)
    m_out, m_req = oracle.epilogue_scales(s_w, s_a, s_a, 1.0, 1, 1)
    acc = oracle.group_conv(q, wq, 1, 1).reshape(-1, G * Co)
    a_ref, y_ref, q_ref = oracle.epilogue(acc, G, m_out, m_req, 1, 1, None, None, True, 2)
    d = B.layer_desc(N, H, W, G, Ci, Co, 3, 1, 1, 2, bits_w, 2, 1, code_format=fmt)
    wp = torch.from_numpy(B.palquant_pack_weights_odd_host(w, d, u)).cuda()
    qd = torch.empty(x.size, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(torch.from_numpy(x).cuda(), qd, N, H, W, G, Ci, 2, inv_s, code_format=fmt)
    ad = torch.empty((N * H * W, G * Co), dtype=torch.int32, device="cuda")
    yd = torch.empty((N * H * W, G * Co), dtype=torch.float32, device="cuda")
    qo = torch.empty(N * H * W * G * Co, dtype=torch.uint8, device="cuda")
    B.palquant_layer_fused(qd, wp, d, m_out, m_req, B.shuffle(1, 1), None, ad, yd, qo)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(ad.cpu().numpy(), a_ref)
    assert np.array_equal(yd.cpu().numpy(), y_ref)
    assert np.array_equal(from_format(qo.cpu().numpy(), fmt, N, H, W, G * Co).reshape(-1, G * Co), q_ref)


# --------------------------- packed FP4 codes (format 4, block-scaled FP4 MMA)
F4_CASES = [
    Case(1, 28, 28, 2, 64, 32, 3, 1, 1, seed=80),
    Case(2, 13, 11, 3, 64, 96, 3, 1, 1, seed=81),                     # odd sizes, six 16-column chunks
    Case(3, 9, 17, 4, 64, 64, 3, 2, 1, seed=82),                      # stride 2 (staged window split into phases)
    Case(2, 10, 10, 2, 64, 128, 1, 2, 0, kind=0, relu=False, seed=83),  # 1x1 stride-2 downsample
    Case(2, 7, 9, 4, 128, 96, 1, 1, 0, seed=84),                      # flat mode, ragged last tile
    Case(2, 14, 14, 8, 64, 32, 3, 1, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=85),
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, seed=86),                   # two output-channel blocks of 128
    Case(1, 7, 7, 2, 1024, 32, 3, 1, 1, seed=87),                     # two K blocks, whole-image tiles
    Case(2, 8, 8, 2, 64, 320, 3, 1, 1, seed=88),                      # 80-column blocks: half-row stores
    Case(1, 5, 130, 1, 64, 32, 3, 1, 1, seed=89),                     # rows wider than 128 positions
    Case(2, 11, 10, 2, 64, 64, 3, 1, 1, shortcut=True, seed=90),      # shortcut add before ReLU
    Case(1, 9, 11, 2, 64, 64, 5, 1, 2, seed=91),                      # 5x5 kernel
    Case(2, 6, 6, 2, 64, 32, 3, 1, 1, bits_out=1, relu=False, kind=1, shift=-1, seed=92),
    Case(1, 16, 16, 4, 64, 64, 3, 2, 0, seed=93),                     # stride 2 without padding
    Case(2, 8, 8, 2, 256, 256, 3, 1, 1, seed=94),                     # 256 channels per group
    Case(1, 10, 10, 2, 192, 64, 3, 1, 1, seed=95),                    # three K steps per tap
    Case(2, 36, 40, 2, 64, 64, 3, 1, 1, shortcut=True, seed=96),      # three accumulators per tile
    Case(1, 40, 30, 2, 64, 64, 3, 2, 1, seed=97),                     # three accumulators, stride 2
    Case(2, 20, 42, 2, 128, 64, 3, 1, 1, seed=98),                    # three accumulators, two K steps
    Case(2, 20, 20, 2, 64, 64, 1, 1, 0, seed=99),                     # flat, two boxes per tile
    Case(2, 17, 17, 2, 128, 64, 1, 1, 0, seed=100),                   # flat, second box wholly past the image
    Case(1, 6, 140, 2, 64, 32, 3, 2, 1, seed=101),                    # stride 2, window wider than one TMA box row
]


@pytest.mark.parametrize("c", F4_CASES, ids=str)
def test_layer_fused_fp4_codes_matches_oracle(B, c):
    ref = prepare(c)
    got = run_gpu(c, ref, fmt=B.PQ_CODES_C32F4)
    assert_layer_parity(c, ref, got)


@pytest.mark.parametrize("c", F4_CASES, ids=str)
def test_layer_codes_only_fp4_matches_oracle(B, c):
    ref = prepare(c)
    got = run_gpu(c, ref, outputs=("q",), fmt=B.PQ_CODES_C32F4)
    assert_layer_parity(c, ref, got)


F4_FULL = [(n, c) for n, c in FULL if c.bits_a <= 2 and c.Cin_g % 64 == 0 and c.Cout_g % 32 == 0]


@pytest.mark.parametrize("name,cfg", F4_FULL, ids=[n for n, _ in F4_FULL])
def test_full_size_codes_only_fp4_sampled(B, name, cfg):
    c = Case(cfg.N, cfg.H, cfg.W, cfg.G, cfg.Cin_g, cfg.Cout_g, cfg.k, cfg.stride, cfg.pad, bits=cfg.bits_a,
             kind=cfg.shuffle_kind, shift=cfg.shuffle_shift, relu=cfg.relu, seed=0)
    pix = _sample_pixels(c.N, c.Ho, c.Wo, 3000, 4)
    ref = prepare(c, sample_pix=pix)
    got = run_gpu(c, ref, outputs=("q",), fmt=B.PQ_CODES_C32F4)
    assert_layer_parity(c, ref, got, pix)


@pytest.mark.parametrize("bits_w,Cin", [(3, 1024), (2, 1024), (3, 64)])
def test_fp4_worst_case_magnitudes_exact(B, bits_w, Cin):
    """Activation codes all 3, weight codes all at an extreme (-4 with 3 bits): the
    largest sums the FP4 path can produce, exact."""
    G, Co, k, N, H, W = 2, 32, 3, 1, 6, 6
    from layer_cases import to_format

    q = np.full((N, H, W, G * Cin), 3, dtype=np.uint8)
    wq = np.full((G, Co, k, k, Cin), -(1 << (bits_w - 1)), dtype=np.int8)
    wq[1] = (1 << (bits_w - 1)) - 1
    d = B.layer_desc(N, H, W, G, Cin, Co, k, 1, 1, 2, bits_w, 2, code_format=B.PQ_CODES_C32F4)
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).cuda()
    acc = torch.zeros((N, H, W, G * Co), dtype=torch.int32, device="cuda")
    B.palquant_group_conv(torch.from_numpy(to_format(q, 4)).cuda(), wp, acc, d)
    assert B.palquant_sync_check() == B.PQ_OK
    ref = oracle.group_conv(q, wq, 1, 1)
    assert np.abs(ref).max() == 9 * Cin * 3 * (1 << (bits_w - 1))
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)


@pytest.mark.parametrize("shape,G,bits", [((2, 7, 9, 64), 4, 2), ((1, 5, 6, 96), 3, 1), ((2, 11, 13, 768), 4, 2),
                                          ((3, 4, 5, 32), 2, 2)])
def test_quantize_act_fp4_matches_oracle(B, shape, G, bits):
    from layer_cases import c32f4_to_nhwc

    gen = synth.generator(sum(shape) + 13)
    x = synth.normal(shape, gen, 2.0)
    x.reshape(-1)[:6] = np.array([0.5, 1.5, 2.5, np.nan, np.inf, -np.inf], dtype=np.float32)
    inv = (synth.half_normal((G,), gen) + 0.5).astype(np.float32)
    q = torch.full((int(np.prod(shape)) // 2,), 254, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(torch.from_numpy(x).cuda(), q, shape[0], shape[1], shape[2], G, shape[3] // G, bits, inv,
                            code_format=B.PQ_CODES_C32F4)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(c32f4_to_nhwc(q.cpu().numpy(), *shape), oracle.quantize_act(x, G, bits, inv))


def test_layer_fp4_with_odd_weight_levels_matches_oracle(B):
    from layer_cases import from_format

    N, H, W, G, Ci, Co = 2, 12, 10, 2, 64, 64
    gen = synth.generator(75)
    x = synth.half_normal((N, H, W, G * Ci), gen)
    w = synth.he_weights(G, Co, 3, 3, Ci, gen)
    s_a = oracle.act_step(x, G, 2)
    inv_s = oracle.inv_step(s_a)
    u = (2.0 * np.abs(w).reshape(G, -1).mean(axis=1)).astype(np.float32)
    s_w = (u.astype(np.float64) / 3.0).astype(np.float32)
    q = oracle.quantize_act(x, G, 2, inv_s)
    wq = oracle.quantize_weights_odd(w, 2, u)
    m_out, m_req = oracle.epilogue_scales(s_w, s_a, s_a, 1.0, 1, 1)
    acc = oracle.group_conv(q, wq, 1, 1).reshape(-1, G * Co)
    a_ref, y_ref, q_ref = oracle.epilogue(acc, G, m_out, m_req, 1, 1, None, None, True, 2)
    d = B.layer_desc(N, H, W, G, Ci, Co, 3, 1, 1, 2, 2, 2, 1, code_format=B.PQ_CODES_C32F4)
    wp = torch.from_numpy(B.palquant_pack_weights_odd_host(w, d, u)).cuda()
    qd = torch.empty(x.size // 2, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act(torch.from_numpy(x).cuda(), qd, N, H, W, G, Ci, 2, inv_s, code_format=B.PQ_CODES_C32F4)
    ad = torch.empty((N * H * W, G * Co), dtype=torch.int32, device="cuda")
    yd = torch.empty((N * H * W, G * Co), dtype=torch.float32, device="cuda")
    qo = torch.empty(N * H * W * G * Co // 2, dtype=torch.uint8, device="cuda")
    B.palquant_layer_fused(qd, wp, d, m_out, m_req, B.shuffle(1, 1), None, ad, yd, qo)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(ad.cpu().numpy(), a_ref)
    assert np.array_equal(yd.cpu().numpy(), y_ref)
    assert np.array_equal(from_format(qo.cpu().numpy(), 4, N, H, W, G * Co).reshape(-1, G * Co), q_ref)


# ------------------------------- quantiser fused into the layer (fp32 in, codes out)
QF_CASES = [
    Case(1, 28, 28, 2, 32, 32, 3, 1, 1, seed=110),                    # config 0 shape
    Case(2, 13, 11, 3, 32, 48, 3, 1, 1, seed=111),                    # odd sizes, three output chunks
    Case(2, 7, 9, 4, 96, 96, 1, 1, 0, seed=112),                      # flat, ragged last tile
    Case(2, 20, 20, 2, 64, 64, 1, 1, 0, seed=113),                    # flat, several tiles
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, seed=114),                  # four K blocks, two output blocks
    Case(1, 7, 7, 2, 256, 32, 3, 1, 1, seed=115),                     # eight K blocks, whole-image tiles
    Case(2, 11, 10, 2, 64, 64, 3, 1, 1, shortcut=True, seed=116),     # shortcut add before ReLU
    Case(1, 9, 11, 2, 32, 64, 5, 1, 2, seed=117),                     # 5x5 kernel
    Case(1, 16, 16, 1, 32, 16, 3, 1, 0, bits=4, kind=0, seed=118),    # pad 0, G = 1, 4-bit
    Case(2, 14, 14, 8, 32, 32, 3, 1, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=119),
    Case(2, 6, 6, 2, 32, 32, 3, 1, 1, bits=3, bits_out=4, relu=False, kind=1, shift=-1, seed=120),
    Case(1, 5, 130, 1, 32, 16, 3, 1, 1, seed=121),                    # rows wider than 128 positions
    Case(2, 36, 40, 2, 64, 64, 3, 1, 1, seed=122),                    # several row tiles per image
]


def _run_quant_fused(B, c, ref, fmt, outputs=("acc", "y", "q")):
    from layer_cases import code_bytes, from_format

    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad, c.bits, c.bits, c.bo, int(c.relu),
                     code_format=fmt)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    B.palquant_pack_weights(ref["w"], d, ref["inv_sw"], wp, nbytes)
    shape = (c.N, c.Ho, c.Wo, c.G * c.Cout)
    acc = torch.full(shape, -7, dtype=torch.int32, device="cuda") if "acc" in outputs else None
    y = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda") if "y" in outputs else None
    qo = torch.full((code_bytes(int(np.prod(shape)), fmt),), 255, dtype=torch.uint8, device="cuda")
    sc = None if ref["shortcut"] is None else torch.from_numpy(ref["shortcut"]).cuda()
    B.palquant_quantize_layer_fused(torch.from_numpy(ref["x"]).cuda(), ref["inv_s"], wp, d, ref["m_out"],
                                    ref["m_req"], B.shuffle(c.kind, c.shift, c.perm), sc, acc, y, qo)
    st = B.palquant_sync_check()
    assert st == B.PQ_OK, B.strerror(st)
    out = dict(q=ref["q"])  # the input codes never leave the kernel
    if acc is not None:
        out["acc"] = acc.cpu().numpy().reshape(-1, c.G * c.Cout)
    if y is not None:
        out["y"] = y.cpu().numpy().reshape(-1, c.G * c.Cout)
    out["q_out"] = from_format(qo.cpu().numpy(), fmt, c.N, c.Ho, c.Wo, c.G * c.Cout).reshape(-1, c.G * c.Cout)
    return out


@pytest.mark.parametrize("fmt", FORMATS, ids=["nhwc", "c16"])
@pytest.mark.parametrize("c", QF_CASES, ids=str)
def test_quantize_layer_fused_matches_oracle(B, c, fmt):
    """Quantise-on-load: the same int32 sums, fp32 outputs and codes as the oracle's
    quantiser followed by its layer."""
    ref = prepare(c)
    assert_layer_parity(c, ref, _run_quant_fused(B, c, ref, fmt))


@pytest.mark.parametrize("c,fmt", [(QF_CASES[0], 2), (QF_CASES[2], 2), (QF_CASES[12], 0), (QF_CASES[4], 2),
                                   (Case(2, 36, 40, 2, 64, 64, 3, 1, 1, seed=136), 4)], ids=str)
def test_quantize_layer_fused_inputs_ready_overlapped(B, c, fmt):
    """PQ_LAYER_INPUTS_READY: back-to-back launches over independent inputs, each one's
    loads starting while the previous launch still runs; two output buffers written
    in turn, so every store must also wait for the launch before (the last two
    launches' codes are checked).  Results equal single flagless launches bit for bit
    and the oracle's codes."""
    from layer_cases import code_bytes, from_format

    from paper_2208_01944_gb300 import synth

    r0 = prepare(c)
    x_np = [r0["x"]] + [synth.half_normal(r0["x"].shape, synth.generator(c.seed + 1000 * i)) for i in range(1, 5)]
    kw = dict(code_format=fmt)
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad, c.bits, c.bits, c.bo, int(c.relu), **kw)
    dr = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad, c.bits, c.bits, c.bo, int(c.relu),
                      flags=B.PQ_LAYER_INPUTS_READY, **kw)
    # one weight set and one set of steps for all launches (those of the first input)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    B.palquant_pack_weights(r0["w"], d, r0["inv_sw"], wp, nbytes)
    shape = (c.N, c.Ho, c.Wo, c.G * c.Cout)
    n_out = code_bytes(int(np.prod(shape)), fmt)
    xs = [torch.from_numpy(x).cuda() for x in x_np]
    shuf = B.shuffle(c.kind, c.shift, c.perm)
    sc = None if r0["shortcut"] is None else torch.from_numpy(r0["shortcut"]).cuda()

    def launch(x, desc, out):
        B.palquant_quantize_layer_fused(x, r0["inv_s"], wp, desc, r0["m_out"], r0["m_req"], shuf, sc, None, None, out)

    outs = [torch.full((n_out,), 255, dtype=torch.uint8, device="cuda") for _ in range(2)]
    for i, x in enumerate(xs):
        launch(x, dr, outs[i % 2])
    assert B.palquant_sync_check() == B.PQ_OK
    for i in (3, 4):
        single = torch.full((n_out,), 255, dtype=torch.uint8, device="cuda")
        launch(xs[i], d, single)
        assert B.palquant_sync_check() == B.PQ_OK
        assert torch.equal(outs[i % 2], single), i
        # against the oracle: input i quantised with the first input's steps, the same layer
        q = oracle.quantize_act(x_np[i], c.G, c.bits, r0["inv_s"])
        acc = oracle.group_conv(q, oracle.quantize_weights(r0["w"], c.bits, r0["inv_sw"]), c.stride, c.pad)
        _, _, q_ref = oracle.epilogue(acc.reshape(-1, c.G * c.Cout), c.G, r0["m_out"], r0["m_req"], c.kind, c.shift,
                                      c.perm, None if sc is None else r0["shortcut"].reshape(-1, c.G * c.Cout),
                                      c.relu, c.bo)
        got = from_format(single.cpu().numpy(), fmt, c.N, c.Ho, c.Wo, c.G * c.Cout).reshape(-1, c.G * c.Cout)
        assert np.array_equal(got, q_ref), i


def test_inputs_ready_chain_reads_output_two_launches_back(B):
    """PQ_LAYER_INPUTS_READY over a chain L1 -> L2 -> L3 in which L2 reads nothing L1
    writes but L3 reads L1's output codes.  L1 fills every SM; L2 is a few CTAs, so
    its CTAs start while most of L1 still runs.  Each layer kernel lets its
    dependent launch start only after its own wait for the kernel before it, so
    L3's early loads cannot start before L1 has completed.  L3's codes equal the
    oracle's layer over the oracle's L1 codes, three chains in a row."""
    from layer_cases import from_format

    fmt = B.PQ_CODES_C16
    c1 = Case(16, 56, 56, 2, 32, 64, 3, 1, 1, seed=140)
    c2 = Case(1, 8, 8, 2, 32, 64, 3, 1, 1, seed=141)
    r1, r2 = prepare(c1), prepare(c2)
    G, C3 = 2, 32
    gen = synth.generator(142)
    w3 = synth.he_weights(G, C3, 3, 3, c1.Cout, gen)
    inv_sw3 = oracle.inv_step(oracle.weight_step(w3, 2))
    s_a3 = np.full(G, 0.75, np.float32)
    m_out3, m_req3 = oracle.epilogue_scales(oracle.weight_step(w3, 2), s_a3, s_a3, 1.0, 1, 1)
    q1_ref = r1["q_ref"].reshape(c1.N, c1.Ho, c1.Wo, G * c1.Cout)
    acc3 = oracle.group_conv(q1_ref, oracle.quantize_weights(w3, 2, inv_sw3), 1, 1).reshape(-1, G * C3)
    _, _, q3_ref = oracle.epilogue(acc3, G, m_out3, m_req3, 1, 1, None, None, True, 2)

    def desc(c, cin, cout, flags):  # 3x3, stride 1, pad 1: the output has the input's size
        return B.layer_desc(c.N, c.H, c.W, G, cin, cout, 3, 1, 1, 2, 2, 2, 1, code_format=fmt, flags=flags)

    d1 = desc(c1, c1.Cin, c1.Cout, 0)
    d2 = desc(c2, c2.Cin, c2.Cout, B.PQ_LAYER_INPUTS_READY)
    d3 = desc(c1, c1.Cout, C3, B.PQ_LAYER_INPUTS_READY)
    wps = []
    for d, w, inv in ((d1, r1["w"], r1["inv_sw"]), (d2, r2["w"], r2["inv_sw"]), (d3, w3, inv_sw3)):
        nb = B.palquant_packed_weight_bytes(d)
        wp = torch.empty(nb, dtype=torch.uint8, device="cuda")
        B.palquant_pack_weights(w, d, inv, wp, nb)
        wps.append(wp)
    x1, x2 = torch.from_numpy(r1["x"]).cuda(), torch.from_numpy(r2["x"]).cuda()
    shuf = B.shuffle(1, 1)
    n1 = c1.N * c1.Ho * c1.Wo * G * c1.Cout
    o2 = torch.empty(c2.N * c2.Ho * c2.Wo * G * c2.Cout, dtype=torch.uint8, device="cuda")
    for rep in range(3):
        o1 = torch.full((n1,), 255, dtype=torch.uint8, device="cuda")
        o3 = torch.full((c1.N * c1.Ho * c1.Wo * G * C3,), 255, dtype=torch.uint8, device="cuda")
        B.palquant_quantize_layer_fused(x1, r1["inv_s"], wps[0], d1, r1["m_out"], r1["m_req"], shuf, None, None,
                                        None, o1)
        B.palquant_quantize_layer_fused(x2, r2["inv_s"], wps[1], d2, r2["m_out"], r2["m_req"], shuf, None, None,
                                        None, o2)
        B.palquant_layer_fused(o1, wps[2], d3, m_out3, m_req3, shuf, None, None, None, o3)
        assert B.palquant_sync_check() == B.PQ_OK
        got1 = from_format(o1.cpu().numpy(), fmt, c1.N, c1.Ho, c1.Wo, G * c1.Cout)
        assert np.array_equal(got1, q1_ref), rep
        got3 = from_format(o3.cpu().numpy(), fmt, c1.N, c1.Ho, c1.Wo, G * C3).reshape(-1, G * C3)
        assert np.array_equal(got3, q3_ref), rep


QF_F4_CASES = [
    Case(1, 28, 28, 2, 64, 32, 3, 1, 1, seed=130),
    Case(2, 13, 11, 3, 64, 96, 3, 1, 1, seed=131),                    # odd sizes
    Case(2, 7, 9, 4, 128, 96, 1, 1, 0, seed=132),                     # flat, ragged last tile
    Case(1, 12, 12, 2, 128, 256, 3, 1, 1, seed=133),                  # two K blocks, two output blocks
    Case(2, 11, 10, 2, 64, 64, 3, 1, 1, shortcut=True, seed=134),     # shortcut add before ReLU
    Case(2, 14, 14, 8, 64, 32, 3, 1, 1, kind=3, perm=(3, 0, 7, 1, 6, 2, 5, 4), seed=135),
    Case(2, 36, 40, 2, 64, 64, 3, 1, 1, seed=136),                    # several row tiles per image
    Case(2, 6, 6, 2, 64, 32, 3, 1, 1, bits_out=1, relu=False, kind=1, shift=-1, seed=137),
]


@pytest.mark.parametrize("c", QF_F4_CASES, ids=str)
def test_quantize_layer_fused_fp4_matches_oracle(B, c):
    """Quantise-on-load into packed FP4 operands (block-scaled FP4 MMAs), FP4 codes out."""
    ref = prepare(c)
    assert_layer_parity(c, ref, _run_quant_fused(B, c, ref, B.PQ_CODES_C32F4))


@pytest.mark.parametrize("c", QF_CASES, ids=str)
def test_quantize_layer_fused_codes_only(B, c):
    """Channel-blocked codes as the only output: the plan reserves no epilogue
    staging and takes larger tiles than with int32 / fp32 outputs."""
    ref = prepare(c)
    assert_layer_parity(c, ref, _run_quant_fused(B, c, ref, 2, outputs=("q",)))


@pytest.mark.parametrize("c", QF_F4_CASES, ids=str)
def test_quantize_layer_fused_fp4_codes_only(B, c):
    ref = prepare(c)
    assert_layer_parity(c, ref, _run_quant_fused(B, c, ref, B.PQ_CODES_C32F4, outputs=("q",)))


QF_FULL = [(n, c) for n, c in FULL if c.stride == 1]


@pytest.mark.parametrize("fmt", [2, 4], ids=["c16", "fp4"])
@pytest.mark.parametrize("name,cfg", QF_FULL, ids=[n for n, _ in QF_FULL])
def test_full_size_quantize_layer_fused_sampled(B, name, cfg, fmt):
    """The benchmarked step at full size, as the benchmark launches it: fp32
    activations in, the next layer's codes out (codes only), sampled pixels
    against the oracle's quantiser followed by its layer."""
    if fmt == 4 and (cfg.bits_a > 2 or cfg.Cin_g % 64 or cfg.Cout_g % 32 or cfg.shuffle_kind == 2):
        pytest.skip("outside the packed-FP4 format")
    c = Case(cfg.N, cfg.H, cfg.W, cfg.G, cfg.Cin_g, cfg.Cout_g, cfg.k, cfg.stride, cfg.pad, bits=cfg.bits_a,
             kind=cfg.shuffle_kind, shift=cfg.shuffle_shift, relu=cfg.relu, seed=0)
    pix = _sample_pixels(c.N, c.Ho, c.Wo, 3000, 3)
    ref = prepare(c, sample_pix=pix)
    got = _run_quant_fused(B, c, ref, fmt, outputs=("q",))
    assert_layer_parity(c, ref, got, pix)


def test_quantize_layer_fused_special_inputs(B):
    """Inputs exactly on rounding ties, NaN, +-inf and negative values quantise as the
    oracle's quantiser does (NaN -> 0, +inf -> Qp, ties to even)."""
    c = Case(2, 10, 12, 2, 64, 32, 3, 1, 1, bits=2, seed=123)
    ref = prepare(c)
    x = ref["x"].copy()
    flat = x.reshape(-1)
    rng = np.random.default_rng(5)
    idx = rng.choice(flat.size, 400, replace=False)
    inv = ref["inv_s"]
    g_of = (np.arange(flat.size) % (c.G * c.Cin)) // c.Cin
    ties = (rng.integers(0, 4, idx.size) + 0.5).astype(np.float32)
    flat[idx[:200]] = ties[:200] / inv[g_of[idx[:200]]]  # x * inv_s lands on (or next to) a tie
    flat[idx[200:250]] = np.nan
    flat[idx[250:300]] = np.inf
    flat[idx[300:350]] = -np.inf
    flat[idx[350:]] = -rng.random(50).astype(np.float32)
    q = oracle.quantize_act(x, c.G, c.bits, inv)
    wq = ref["wq"]
    acc = oracle.group_conv(q, wq, c.stride, c.pad).reshape(-1, c.G * c.Cout)
    a_ref, y_ref, q_ref = oracle.epilogue(acc, c.G, ref["m_out"], ref["m_req"], c.kind, c.shift, None, None, True, c.bo)
    ref2 = dict(ref, x=x, q=q, acc_ref=a_ref, y_ref=y_ref, q_ref=q_ref)
    assert_layer_parity(c, ref2, _run_quant_fused(B, c, ref2, 2))
