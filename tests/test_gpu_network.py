"""The ResNet-18-shaped PalQuant network on the GPU against the oracle network.

Both sides receive the same seeded images and weights and the oracle's calibrated
steps; every intermediate tensor is compared: full-precision stem and pooling outputs
and logits bit for bit (fixed summation order on both sides), all codes bit for bit,
and the blocks' fp32 outputs bit for bit (one fp32 multiply and one add per value).
"""
import numpy as np
import pytest
import torch

import oracle.resnet as OR
from layer_cases import from_format
from paper_2208_01944_gb300 import synth

pytestmark = pytest.mark.gpu


def _codes(t, fmt):
    N, H, W, C = t.shape
    return from_format(t.cpu().numpy(), fmt, N, H, W, C * (2 if fmt == 4 else 1))


def _compare(net, r):
    f = net.fmt
    if net.stem_out is not None:
        assert np.array_equal(net.stem_out.cpu().numpy(), r["stem"]), "stem"
    assert np.array_equal(net.pool.cpu().numpy(), r["pool"]), "max pooling"
    if not net.fuse_input:  # else the input codes exist only inside the first conv1
        assert np.array_equal(_codes(net.in_codes, f), r[net.blocks[0]["name"] + ".in_codes"]), "input codes"
    for i, blk in enumerate(net.blocks):
        n = blk["name"]
        assert np.array_equal(_codes(blk["mid_codes"], f), r[n + ".mid_codes"]), n + " conv1 codes"
        if blk["down"]:
            assert np.array_equal(blk["down_out"].cpu().numpy(), r[n + ".down"]), n + " downsample"
        assert np.array_equal(blk["out"].cpu().numpy(), r[n + ".out"]), n + " block output"
        if i + 1 < len(net.blocks):
            assert np.array_equal(_codes(blk["out_codes"], f), r[n + ".out_codes"]), n + " next-block codes"
    assert np.array_equal(net.avg.cpu().numpy(), r["avg"]), "average pooling"
    assert np.array_equal(net.logits.cpu().numpy(), r["logits"]), "logits"


@pytest.mark.parametrize("N,H,widths,classes,seed,fmt", [(2, 32, (32, 32, 32, 32), 10, 1, 2),
                                                         (3, 64, (32, 64, 32, 64), 16, 2, 2),
                                                         (2, 48, (64, 64, 128, 64), 12, 4, 4),   # FP4 codes
                                                         (2, 48, (64, 64, 128, 64), 12, 4, 2)])
def test_small_network_matches_oracle(N, H, widths, classes, seed, fmt):
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    x, params = synth.resnet18_inputs(N, H, H, 2, widths, classes, seed=seed)
    steps = OR.calibrate(x, params, 2, 2)
    r = OR.forward(x, params, 2, 2, steps)
    net = PalQuantResNet18(params, N, H, H, 2, widths, classes, 2, code_format=fmt)
    assert net.fmt == fmt
    net.set_steps(steps)
    xd = torch.from_numpy(x).cuda()
    net.forward(xd)
    net.stream.synchronize()
    from paper_2208_01944_gb300 import binding as B
    assert B.palquant_sync_check() == B.PQ_OK
    _compare(net, r)


def test_resnet18_224_matches_oracle():
    """The full ResNet-18 shape (224x224 input, per-group widths 64/128/256/512, G = 2,
    1000 classes) on one image, and the CUDA-graph replay of the same forward."""
    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    x, params = synth.resnet18_inputs(1, seed=0)
    steps = OR.calibrate(x, params, 2, 2)
    r = OR.forward(x, params, 2, 2, steps)
    xd = torch.from_numpy(x).cuda()
    # the default (FP4 nibbles, the stem output kept for the comparison), and one code
    # per byte with the stem output never written
    for fmt, keep in ((B.PQ_CODES_C32F4, True), (B.PQ_CODES_C16, False)):
        net = PalQuantResNet18(params, 1, code_format=None if fmt == B.PQ_CODES_C32F4 else fmt, keep_stem=keep)
        assert net.fused_stem and (net.stem_out is not None) == keep
        assert net.fmt == fmt
        net.set_steps(steps)
        net.forward(xd)
        net.stream.synchronize()
        assert B.palquant_sync_check() == B.PQ_OK
        _compare(net, r)
        net.logits.zero_()
        net.capture(xd)
        net.replay()
        net.stream.synchronize()
        assert B.palquant_sync_check() == B.PQ_OK
        assert np.array_equal(net.logits.cpu().numpy(), r["logits"])
        del net


def test_device_calibration_close_to_oracle():
    """The library's own step initialisation (device sums) on the same network: the
    first block's input steps and every weight step within one float ulp of the oracle's."""
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    x, params = synth.resnet18_inputs(2, 32, 32, 2, (32, 32, 32, 32), 10, seed=3)
    ref = OR.calibrate(x, params, 2, 2)
    net = PalQuantResNet18(params, 2, 32, 32, 2, (32, 32, 32, 32), 10, 2)
    got = net.calibrate(torch.from_numpy(x).cuda())
    assert set(got) == set(ref)
    keys = ["s1b1.in"] + [k for k in ref if k.endswith(".w")]
    for k in keys:
        d = np.abs(got[k].view(np.int32).astype(np.int64) - ref[k].view(np.int32).astype(np.int64))
        assert np.all(d <= 1), k
    for k in ref:
        assert np.allclose(got[k], ref[k], rtol=1e-3), k


# ------------------------------------------------------------ full-precision layers alone
@pytest.mark.parametrize("shape,Cout,k,s,p,relu", [
    ((2, 37, 29, 3), 64, 7, 2, 3, True),     # the stem shape at 64 channels (the generic kernel)
    ((1, 224, 224, 3), 128, 7, 2, 3, True),  # the network's stem shape (the stem kernel)
    ((2, 30, 34, 3), 128, 7, 2, 3, False),   # the stem kernel without ReLU, ragged tiles
    ((2, 9, 11, 5), 32, 3, 1, 1, False),     # the generic kernel, weights in shared memory
    ((1, 12, 10, 64), 48, 5, 2, 2, True),    # the generic kernel, weights from global memory
])
def test_conv2d_f32_matches_oracle(shape, Cout, k, s, p, relu):
    import oracle
    from paper_2208_01944_gb300 import binding as B

    gen = synth.generator(sum(shape) + Cout)
    x = synth.normal(shape, gen)
    w = synth.normal((Cout, k, k, shape[3]), gen, 0.2)
    ref = oracle.conv2d_f32(x, w, s, p, relu)
    y = torch.empty(ref.shape, dtype=torch.float32, device="cuda")
    B.palquant_conv2d_f32(torch.from_numpy(x).cuda(), torch.from_numpy(w).cuda(), y, shape[0], shape[1], shape[2],
                          shape[3], Cout, k, s, p, relu)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(y.cpu().numpy(), ref)


@pytest.mark.parametrize("N,H,W,keep", [(2, 224, 224, True), (2, 37, 29, True), (3, 50, 46, False), (1, 13, 9, True)])
def test_stem_pool_f32_matches_oracle(N, H, W, keep):
    """The fused stem + max pooling: the pooled output (and the stem output when asked
    for) bit for bit against the oracle's separate convolution and pooling; tiles
    ragged at the image's right and bottom edges, and images of one tile."""
    import oracle
    from paper_2208_01944_gb300 import binding as B

    gen = synth.generator(N * 1000 + H + W)
    x = synth.normal((N, H, W, 3), gen)
    w = synth.normal((128, 7, 7, 3), gen, 0.2)
    stem = oracle.conv2d_f32(x, w, 2, 3, True)
    ref = oracle.maxpool_f32(stem, 3, 2, 1)
    pool = torch.full(ref.shape, float("nan"), dtype=torch.float32, device="cuda")  # the call zeroes it
    st = torch.empty(stem.shape, dtype=torch.float32, device="cuda") if keep else None
    B.palquant_stem_pool_f32(torch.from_numpy(x).cuda(), torch.from_numpy(w).cuda(), st, pool, N, H, W, 128)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(pool.cpu().numpy(), ref)
    if keep:
        assert np.array_equal(st.cpu().numpy(), stem)


def test_stem_pool_f32_rejects_other_widths():
    from paper_2208_01944_gb300 import binding as B

    x = torch.zeros((1, 16, 16, 3), device="cuda")
    w = torch.zeros((64, 7, 7, 3), device="cuda")
    pool = torch.empty((1, 4, 4, 64), device="cuda")
    with pytest.raises(RuntimeError):
        B.palquant_stem_pool_f32(x, w, None, pool, 1, 16, 16, 64)


def test_pooling_and_linear_match_oracle():
    import oracle
    from paper_2208_01944_gb300 import binding as B

    gen = synth.generator(21)
    x = synth.normal((3, 13, 11, 24), gen)
    ref = oracle.maxpool_f32(x, 3, 2, 1)
    y = torch.empty(ref.shape, dtype=torch.float32, device="cuda")
    B.palquant_maxpool2d_f32(torch.from_numpy(x).cuda(), y, 3, 13, 11, 24, 3, 2, 1)
    assert np.array_equal(y.cpu().numpy(), ref)
    x5 = synth.normal((2, 7, 9, 5), gen)  # channels not a multiple of 4: the scalar kernel
    ref5 = oracle.maxpool_f32(x5, 3, 2, 1)
    y5 = torch.empty(ref5.shape, dtype=torch.float32, device="cuda")
    B.palquant_maxpool2d_f32(torch.from_numpy(x5).cuda(), y5, 2, 7, 9, 5, 3, 2, 1)
    assert np.array_equal(y5.cpu().numpy(), ref5)
    ref = oracle.avgpool_f32(x)
    y = torch.empty(ref.shape, dtype=torch.float32, device="cuda")
    B.palquant_avgpool_f32(torch.from_numpy(x).cuda(), y, 3, 13, 11, 24)
    assert np.array_equal(y.cpu().numpy(), ref)
    v = synth.normal((13, 100), gen)
    w = synth.normal((1000, 100), gen)
    ref = oracle.linear_f32(v, w)
    y = torch.empty(ref.shape, dtype=torch.float32, device="cuda")
    B.palquant_linear_f32(torch.from_numpy(v).cuda(), torch.from_numpy(w).cuda(), y, 13, 100, 1000)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(y.cpu().numpy(), ref)


def _compare_paper(net, r):
    f = net.fmt
    assert np.array_equal(net.pool.cpu().numpy(), r["pool"]), "max pooling"
    for m in net.modules:
        n = m["name"]
        assert np.array_equal(_codes(m["in_codes"], f), r[n + ".in_codes"]), n + " input codes"
        assert np.array_equal(m["z"].cpu().numpy(), r[n + ".out"]), n + " module output"
        assert np.array_equal(_codes(m["codes"], f), r[n + ".out_codes"]), n + " module codes"
    for blk in net.blocks:
        n = blk["name"]
        assert np.array_equal(_codes(blk["mid_codes"], f), r[n + ".mid_codes"]), n + " conv1 codes"
        if blk["down"]:
            assert np.array_equal(blk["down_out"].cpu().numpy(), r[n + ".down"]), n + " downsample"
        assert np.array_equal(blk["out"].cpu().numpy(), r[n + ".out"]), n + " block output"
        if n + ".out_codes" in r:
            assert np.array_equal(_codes(blk["out_codes"], f), r[n + ".out_codes"]), n + " next-block codes"
    assert np.array_equal(net.logits.cpu().numpy(), r["logits"]), "logits"


@pytest.mark.parametrize("N,H,widths,classes,seed,fmt", [(2, 32, (32, 32, 32, 32), 10, 7, 2),
                                                         (2, 48, (64, 64, 128, 64), 12, 8, 4),   # FP4 codes
                                                         (3, 64, (32, 64, 32, 64), 16, 9, 2)])
def test_paper_placement_matches_oracle(N, H, widths, classes, seed, fmt):
    """Sec. 4.3's placement: a cyclic shuffle module at each stage's start, the channel
    shuffle at each stage's end; every tensor bit for bit against the oracle network."""
    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    x, params = synth.resnet18_inputs(N, H, H, 2, widths, classes, seed=seed, cyclic_modules=True)
    steps = OR.calibrate(x, params, 2, 2, placement="paper")
    r = OR.forward(x, params, 2, 2, steps, placement="paper")
    net = PalQuantResNet18(params, N, H, H, 2, widths, classes, 2, code_format=fmt, placement="paper")
    net.set_steps(steps)
    net.forward(torch.from_numpy(x).cuda())
    net.stream.synchronize()
    assert B.palquant_sync_check() == B.PQ_OK
    _compare_paper(net, r)


def test_paper_placement_gpu_calibration_matches_oracle():
    """The library's step initialisation for the paper placement: the first module's
    input steps and every weight step within one float ulp of the oracle's, the
    later steps (which depend on codes an ulp can flip) within 1e-3."""
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    x, params = synth.resnet18_inputs(2, 32, 32, 2, (32, 32, 32, 32), 10, seed=7, cyclic_modules=True)
    ref = OR.calibrate(x, params, 2, 2, placement="paper")
    net = PalQuantResNet18(params, 2, 32, 32, 2, (32, 32, 32, 32), 10, 2, code_format=2, placement="paper")
    got = net.calibrate(torch.from_numpy(x).cuda())
    assert set(got) == set(ref)
    for k in ["s1.csm.in"] + [k for k in ref if k.endswith(".w")]:
        d = np.abs(got[k].view(np.int32).astype(np.int64) - ref[k].view(np.int32).astype(np.int64))
        assert np.all(d <= 1), k
    for k in ref:
        assert np.allclose(got[k], ref[k], rtol=1e-3), k
