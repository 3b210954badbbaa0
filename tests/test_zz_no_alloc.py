"""palquant_act_steps_noalloc: the step initialisation for callers that cannot
allocate device memory (their memory is owned elsewhere or budgeted up front).

It keeps its scratch in a fixed array inside the library instead of taking a
caller buffer.  It runs the same two kernels as palquant_act_steps over the same
fixed 256-block partition, so its steps must be bit-identical to that entry
point's; this checks that through the C ABI on two calls in a row (the array is
reused between them), checks both against the oracle's steps (a different
summation order, so within one ulp), and checks that a group count beyond the
array's capacity is refused.  The file is named so that pytest collects it last.
"""
import numpy as np
import pytest

import oracle
from paper_2208_01944_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _ulps(a, b):
    return np.abs(a.view(np.int32).astype(np.int64) - b.view(np.int32).astype(np.int64))


def test_noalloc_steps_match_allocating_entry_point_twice():
    assert torch.cuda.is_available(), "GPU test"
    from paper_2208_01944_gb300 import binding as B

    shapes = [((4, 17, 9, 3 * 32), 3, 2), ((2, 11, 13, 8 * 16), 8, 4)]
    for call, (shape, G, bits) in enumerate(shapes):
        gen = synth.generator(100 + call)
        x_np = synth.half_normal(shape, gen)
        x = torch.from_numpy(x_np).cuda()
        N, H, W, C = shape
        nbytes = B.palquant_act_steps_scratch_bytes(N * H * W, G)
        scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        ref = B.palquant_act_steps(x, N, H, W, G, C // G, bits, scratch, nbytes)
        got = B.palquant_act_steps_noalloc(x, N, H, W, G, C // G, bits)
        # same kernels, same partition, same order: identical bits
        assert np.array_equal(got.view(np.int32), ref.view(np.int32)), (call, got, ref)
        # and the steps of Sec. 5's initialisation, summed in another order
        want = oracle.act_step(x_np, G, bits)
        assert np.all(_ulps(got, want) <= 1), (call, got, want)
    assert B.palquant_sync_check() == B.PQ_OK


def test_noalloc_refuses_more_groups_than_its_scratch_holds():
    assert torch.cuda.is_available(), "GPU test"
    from paper_2208_01944_gb300 import binding as B

    x = torch.ones((1, 2, 2, 65), dtype=torch.float32, device="cuda")
    with pytest.raises(B.PalquantError) as e:
        B.palquant_act_steps_noalloc(x, 1, 2, 2, 65, 1, 2)
    assert e.value.status == B.PQ_EUNSUPPORTED
