"""GPU parity of the quantisation-aware training kernels (Sec. 3.2 Eq. 2-3 with
learned bounds l, u; Sec. 5 straight-through estimator) against the oracle:
forward outputs and input gradients bit for bit, the per-group gradients of l and u
within the bound the C-ABI states (1e-6 of c / r^2 * sum |dy (x - bound)|)."""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2208_01944_gb300 import binding
    return binding


def _inputs(P, G, Cg, bits, seed, ties=True, special=True):
    rng = np.random.default_rng(seed)
    l = rng.uniform(-1.0, 0.5, G).astype(np.float32)
    u = (l + rng.uniform(0.25, 3.0, G)).astype(np.float32)
    x = np.empty((P, G * Cg), np.float32)
    for g in range(G):
        span = float(u[g] - l[g])
        x[:, g * Cg:(g + 1) * Cg] = rng.uniform(float(l[g]) - 0.3 * span, float(u[g]) + 0.3 * span, (P, Cg))
    flat = x.reshape(-1)
    if ties and flat.size >= 64:
        # values whose scaled position lands on (or next to) a rounding tie of the forward
        qp = (1 << bits) - 1
        idx = rng.choice(flat.size, flat.size // 8, replace=False)
        g_of = (idx % (G * Cg)) // Cg
        k = rng.integers(0, qp, idx.size) + 0.5
        flat[idx] = (l[g_of] + (k / qp) * (u[g_of] - l[g_of])).astype(np.float32)
    if special and flat.size >= 64:
        idx = rng.choice(flat.size, 16, replace=False)
        flat[idx[:4]] = np.nan
        flat[idx[4:8]] = np.inf
        flat[idx[8:12]] = -np.inf
        flat[idx[12:]] = l[(idx[12:] % (G * Cg)) // Cg]  # exactly on the lower bound: t = 0, outside
    dy = rng.normal(size=x.shape).astype(np.float32)
    return x, dy, l, u


CASES = [  # P, G, Cg, bits, kind
    (1, 1, 4, 2, 0),
    (37, 3, 20, 3, 1),      # ragged: 5 float4s per group row
    (1000, 4, 64, 2, 0),
    (5, 8, 12, 1, 0),
    (1, 2, 4096, 4, 1),     # weights: one row, the group's weights along it
    (333, 2, 32, 8, 0),
    (2048, 1, 4, 2, 1),     # one float4 per row (the unit divisor)
]


def _run(B, x, dy, G, bits, kind, l, u):
    P, C = x.shape
    Cg = C // G
    xd = torch.from_numpy(x).cuda()
    yd = torch.full_like(xd, 7.0)
    B.palquant_fake_quant_forward(xd, yd, P, G, Cg, bits, kind, l, u)
    dyd = torch.from_numpy(dy).cuda()
    dxd = torch.full_like(xd, 7.0)
    dl = torch.full((G,), 7.0, dtype=torch.float64, device="cuda")
    du = torch.full((G,), 7.0, dtype=torch.float64, device="cuda")
    sb = B.palquant_fake_quant_scratch_bytes(P, G, Cg)
    scratch = torch.empty(max(sb, 16), dtype=torch.uint8, device="cuda")
    B.palquant_fake_quant_backward(xd, dyd, dxd, dl, du, P, G, Cg, bits, kind, l, u, scratch, sb)
    torch.cuda.synchronize()
    return yd.cpu().numpy(), dxd.cpu().numpy(), dl.cpu().numpy(), du.cpu().numpy()


def _grad_bound(x, dy, G, kind, l, u, dx_ref):
    """The C-ABI's bound on dl, du: 1e-6 of c / r^2 * sum |dy (x - bound)| over the inside elements."""
    c = 2.0 if kind else 1.0
    Cg = x.shape[1] // G
    bl, bu = np.zeros(G), np.zeros(G)
    for g in range(G):
        xs = x[:, g * Cg:(g + 1) * Cg].astype(np.float64)
        inside = dx_ref[:, g * Cg:(g + 1) * Cg] != 0
        d = dy[:, g * Cg:(g + 1) * Cg].astype(np.float64)
        r = float(u[g]) - float(l[g])
        bl[g] = 1e-6 * c / r ** 2 * np.sum(np.abs(d * (xs - float(u[g])))[inside]) + 1e-300
        bu[g] = 1e-6 * c / r ** 2 * np.sum(np.abs(d * (xs - float(l[g])))[inside]) + 1e-300
    return bl, bu


@pytest.mark.parametrize("P,G,Cg,bits,kind", CASES)
def test_fake_quant_matches_oracle(B, P, G, Cg, bits, kind):
    x, dy, l, u = _inputs(P, G, Cg, bits, seed=P + 7 * G + Cg + bits)
    y, dx, dl, du = _run(B, x, dy, G, bits, kind, l, u)
    y_ref = oracle.fake_quant_forward(x, G, bits, kind, l, u)
    dx_ref, dl_ref, du_ref = oracle.fake_quant_backward(x, dy, G, bits, kind, l, u)
    assert np.array_equal(y, y_ref, equal_nan=True)
    assert np.array_equal(dx, dx_ref, equal_nan=True)
    bl, bu = _grad_bound(x, dy, G, kind, l, u, dx_ref)
    assert np.all(np.abs(dl - dl_ref) <= bl), (dl, dl_ref)
    assert np.all(np.abs(du - du_ref) <= bu), (du, du_ref)


def test_fake_quant_gradients_deterministic_and_empty(B):
    x, dy, l, u = _inputs(4096, 4, 64, 2, seed=3)
    a = _run(B, x, dy, 4, 2, 0, l, u)
    b = _run(B, x, dy, 4, 2, 0, l, u)
    assert np.array_equal(a[2], b[2]) and np.array_equal(a[3], b[3])
    # no elements: zero gradients
    _, _, dl, du = _run(B, np.zeros((0, 8), np.float32), np.zeros((0, 8), np.float32), 2, 2, 0, l[:2], u[:2])
    assert np.all(dl == 0) and np.all(du == 0)


def test_fake_quant_full_size_activations(B):
    """The benchmarked activation tensor (64x56x56x256 fp32, G = 4): every output and
    input gradient, the group gradients within the bound."""
    from paper_2208_01944_gb300 import workloads
    c = workloads.CONFIG1
    P, G, Cg = c.N * c.H * c.W, c.G, c.Cin_g
    x, dy, l, u = _inputs(P, G, Cg, c.bits_a, seed=11, special=False)
    y, dx, dl, du = _run(B, x, dy, G, c.bits_a, 0, l, u)
    y_ref = oracle.fake_quant_forward(x, G, c.bits_a, 0, l, u)
    dx_ref, dl_ref, du_ref = oracle.fake_quant_backward(x, dy, G, c.bits_a, 0, l, u)
    assert np.array_equal(y, y_ref)
    assert np.array_equal(dx, dx_ref)
    bl, bu = _grad_bound(x, dy, G, 0, l, u, dx_ref)
    assert np.all(np.abs(dl - dl_ref) <= bl) and np.all(np.abs(du - du_ref) <= bu)
