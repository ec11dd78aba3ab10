"""The failure path of the decode kernel on the GPU, with nothing faulted, trapped or hung:
one consumer warp's bounded wait is made to expire (a shared-memory barrier that nothing
completes and no copy targets, limited to a few milliseconds).  The launch must still end
with the product correct, sp_check must report SP_ERR_TIMEOUT once (and clear it), and the
next ordinary calls on the same workspace must be correct against the float64 oracle."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape,M", [((1000, 1024), 1), ((4096, 4096), 4)])
def test_expired_wait_is_reported_and_the_next_call_is_correct(oracle, shape, M):
    import time

    import torch

    from paper_2405_03594_gb300 import sp

    N, K = shape
    g = np.random.default_rng(N + M)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, 70)
    x = synth.activations(M, K, g)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    assert h.kernel_name(M) == "linear_ccw_kernel"
    xd = gu.bf16_to_dev(x)
    ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device="cuda")
    y = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    sp.check()
    t0 = time.perf_counter()
    h.test_expired_wait(xd, y, ws, wait_ms=20)
    with pytest.raises(sp.SpError) as e:
        sp.check()
    assert e.value.code == 6  # SP_ERR_TIMEOUT
    assert time.perf_counter() - t0 < 5.0  # the launch ended after the one expired wait
    sp.check()  # reported once, then cleared
    ref = oracle.linear_bf16(x, W, mask)
    gu.assert_close(gu.bf16_from_dev(y), ref, f"the launch with the expired wait {N}x{K} M={M}")
    for _ in range(2):
        y2 = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
        h.linear(xd, out=y2, workspace=ws)
        sp.check()
        gu.assert_close(gu.bf16_from_dev(y2), ref, f"after the expired wait {N}x{K} M={M}")


def test_expired_wait_argument_checks():
    import torch

    from paper_2405_03594_gb300 import sp

    W = synth.weight(300, 256, np.random.default_rng(1))
    mask = synth.magnitude_mask(W, 70)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    ws = torch.zeros(max(h.workspace_size(5), 256), dtype=torch.uint8, device="cuda")
    x5 = torch.zeros((5, 256), dtype=torch.bfloat16, device="cuda")
    y5 = torch.empty((5, 300), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sp.SpError) as e:
        h.test_expired_wait(x5, y5, ws, 10)  # m outside 1..4
    assert e.value.code == 2
    with pytest.raises(sp.SpError) as e:
        h.test_expired_wait(x5[:1], y5[:1], ws, 0)  # wait_ms outside 1..10000
    assert e.value.code == 1
    sp.check()
