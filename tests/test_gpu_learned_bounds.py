"""GPU parity of the inference quantisers with learned bounds l < u (Sec. 3.2 Eq. 2 as
the paper trains it): the standalone quantiser in every code format and the quantiser
fused into the layer, against the oracle's codes (the training forward's x_q), the
oracle's group convolution and epilogue, bit for bit.  Negative lower bounds check
that the zero padding stays code 0 in the fused form."""
import numpy as np
import pytest

import oracle
from layer_cases import Case, assert_layer_parity, code_bytes, from_format
from paper_2208_01944_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2208_01944_gb300 import binding
    return binding


def _bounds(G, seed, negative=True):
    rng = np.random.default_rng(seed)
    l = rng.uniform(-0.8 if negative else 0.05, 0.3, G).astype(np.float32)
    u = (l + rng.uniform(0.5, 3.0, G)).astype(np.float32)
    return l, u


def _x(shape, G, l, u, bits, seed):
    """Values spread over [l - 0.3 r, u + 0.3 r] per group, an eighth on rounding ties,
    and a few NaN / inf."""
    rng = np.random.default_rng(seed)
    C = shape[-1]
    Cg = C // G
    x = np.empty(shape, np.float32)
    for g in range(G):
        r = float(u[g] - l[g])
        x[..., g * Cg:(g + 1) * Cg] = rng.uniform(float(l[g]) - 0.3 * r, float(u[g]) + 0.3 * r,
                                                   shape[:-1] + (Cg,))
    flat = x.reshape(-1)
    qp = (1 << bits) - 1
    idx = rng.choice(flat.size, flat.size // 8, replace=False)
    g_of = (idx % C) // Cg
    k = rng.integers(0, qp, idx.size) + 0.5
    flat[idx] = (l[g_of] + (k / qp) * (u[g_of] - l[g_of])).astype(np.float32)
    sp = rng.choice(flat.size, min(12, flat.size), replace=False)
    flat[sp[:4]] = np.nan
    flat[sp[4:8]] = np.inf
    flat[sp[8:]] = -np.inf
    return x


@pytest.mark.parametrize("fmt,shape,G,bits", [
    (0, (2, 7, 9, 64), 2, 2),     # NHWC, 16-element vectors
    (0, (1, 5, 6, 30), 3, 3),     # NHWC, any shape (scalar path)
    (2, (2, 9, 11, 96), 3, 4),    # channel-blocked bytes
    (3, (1, 8, 8, 64), 2, 2),     # packed 2-bit words
    (4, (2, 6, 10, 128), 2, 2),   # FP4 nibbles
    (2, (64, 56, 56, 256), 4, 2),  # the benchmarked activation tensor
])
def test_quantize_act_lu_matches_oracle(B, fmt, shape, G, bits):
    N, H, W, C = shape
    l, u = _bounds(G, seed=C + bits)
    x = _x(shape, G, l, u, bits, seed=N + H)
    ref = oracle.quantize_act_lu(x, G, bits, l, u)
    q = torch.full((code_bytes(x.size, fmt),), 0xA5, dtype=torch.uint8, device="cuda")
    B.palquant_quantize_act_lu(torch.from_numpy(x).cuda(), q, N, H, W, G, C // G, bits, l, u, code_format=fmt)
    assert B.palquant_sync_check() == B.PQ_OK
    got = q.cpu().numpy()
    got = got.reshape(shape) if fmt == 0 else from_format(got, fmt, N, H, W, C)
    assert np.array_equal(got, ref)


LU_CASES = [  # the layer shapes of the quantise-on-load cases; l < 0 in all but one
    (Case(1, 28, 28, 2, 32, 32, 3, 1, 1, seed=140), 2, True),
    (Case(2, 13, 11, 3, 32, 48, 3, 1, 1, seed=141), 2, True),
    (Case(2, 7, 9, 4, 96, 96, 1, 1, 0, seed=142), 2, True),       # flat, ragged last tile
    (Case(1, 12, 12, 2, 128, 256, 3, 1, 1, seed=143), 2, True),   # several K blocks and output blocks
    (Case(2, 11, 10, 2, 64, 64, 3, 1, 1, shortcut=True, seed=144), 2, False),
    (Case(2, 14, 14, 2, 64, 64, 3, 1, 1, bits=3, seed=145), 2, True),
    (Case(2, 13, 11, 3, 64, 96, 3, 1, 1, seed=146), 4, True),     # FP4 operands and codes
    (Case(2, 36, 40, 2, 64, 64, 3, 1, 1, seed=147), 4, True),     # several row tiles per image
]


@pytest.mark.parametrize("c,fmt,negative", LU_CASES, ids=lambda v: str(v) if isinstance(v, Case) else str(v))
def test_quantize_layer_fused_lu_matches_oracle(B, c, fmt, negative):
    G = c.G
    l, u = _bounds(G, seed=c.seed, negative=negative)
    gen = synth.generator(c.seed)
    w = synth.he_weights(G, c.Cout, c.k, c.k, c.Cin, gen)
    x = _x((c.N, c.H, c.W, G * c.Cin), G, l, u, c.bits, seed=c.seed + 1)
    s_w = oracle.weight_step(w, c.bits)
    inv_sw = oracle.inv_step(s_w)
    q = oracle.quantize_act_lu(x, G, c.bits, l, u)
    wq = oracle.quantize_weights(w, c.bits, inv_sw)
    acc = oracle.group_conv(q, wq, c.stride, c.pad).reshape(-1, G * c.Cout)
    # de-quantised activations are x_q / (2^b - 1): the layer's scale is s_w / Qp per group
    qp = (1 << c.bits) - 1
    s_a = np.full(G, 1.0 / qp, np.float32)
    m_out, _ = oracle.epilogue_scales(s_w, s_a, None, 1.0, c.kind, c.shift, c.perm)
    _, y0, _ = oracle.epilogue(acc, G, m_out, None, c.kind, c.shift, c.perm, None, True, c.bo)
    s_next = np.maximum(2.0 * y0.reshape(-1, G, c.Cout).astype(np.float64).mean(axis=(0, 2)), 1e-3).astype(np.float32)
    m_out, m_req = oracle.epilogue_scales(s_w, s_a, s_next, 1.0, c.kind, c.shift, c.perm)
    sc = synth.normal((c.N, c.Ho, c.Wo, G * c.Cout), gen) if c.shortcut else None
    a_ref, y_ref, q_ref = oracle.epilogue(acc, G, m_out, m_req, c.kind, c.shift, c.perm,
                                          None if sc is None else sc.reshape(-1, G * c.Cout), c.relu, c.bo)
    d = B.layer_desc(c.N, c.H, c.W, G, c.Cin, c.Cout, c.k, c.stride, c.pad, c.bits, c.bits, c.bo, int(c.relu),
                     code_format=fmt)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    B.palquant_pack_weights(w, d, inv_sw, wp, nbytes)
    shape = (c.N, c.Ho, c.Wo, G * c.Cout)
    xd = torch.from_numpy(x).cuda()
    scd = None if sc is None else torch.from_numpy(sc).cuda()
    # all outputs, then codes only (the plan without epilogue staging)
    acc_d = torch.full(shape, -7, dtype=torch.int32, device="cuda")
    y_d = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
    qo = torch.full((code_bytes(int(np.prod(shape)), fmt),), 255, dtype=torch.uint8, device="cuda")
    shuf = B.shuffle(c.kind, c.shift, c.perm)
    B.palquant_quantize_layer_fused_lu(xd, l, u, wp, d, m_out, m_req, shuf, scd, acc_d, y_d, qo)
    qo2 = torch.full_like(qo, 255)
    B.palquant_quantize_layer_fused_lu(xd, l, u, wp, d, m_out, m_req, shuf, scd, None, None, qo2)
    assert B.palquant_sync_check() == B.PQ_OK
    got = dict(q=q, acc=acc_d.cpu().numpy().reshape(-1, G * c.Cout), y=y_d.cpu().numpy().reshape(-1, G * c.Cout),
               q_out=from_format(qo.cpu().numpy(), fmt, c.N, c.Ho, c.Wo, G * c.Cout).reshape(-1, G * c.Cout))
    ref = dict(q=q, acc_ref=a_ref, y_ref=y_ref, q_ref=q_ref, m_out=m_out)
    assert_layer_parity(c, ref, got)
    q2 = from_format(qo2.cpu().numpy(), fmt, c.N, c.Ho, c.Wo, G * c.Cout).reshape(-1, G * c.Cout)
    assert np.array_equal(q2, q_ref)


def test_learned_bounds_argument_rules(B):
    x = torch.zeros((1, 4, 4, 32), device="cuda")
    q = torch.zeros((1, 4, 4, 32), dtype=torch.uint8, device="cuda")
    for l, u in (([0.0, 1.0], [1.0, 1.0]), ([0.0, float("nan")], [1.0, 2.0]), ([0.0, 0.0], [1.0, float("inf")])):
        with pytest.raises(B.PalquantError) as e:
            B.palquant_quantize_act_lu(x, q, 1, 4, 4, 2, 16, 2, l, u)
        assert e.value.status == B.PQ_EINVAL
