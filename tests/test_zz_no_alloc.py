"""sp_linear_noalloc -- for callers that cannot allocate device memory (for example code
handed only its input and output buffers by a framework that owns every allocation, or a
latency-critical loop where cudaMalloc/cudaFree would synchronise the device) -- must give
the same results as sp_linear through the C ABI, call after call, using the library's
static scratch array instead of a caller workspace, and match the float64 oracle within the
acceptance tolerances; batches above 16 rows take several launches that share the array.

Collected last on purpose: it runs on its own in a fresh process and after every other test."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape,pct,M", [((1000, 1024), 70, 1), ((4096, 4096), 70, 4), ((22016, 4096), 70, 16),
                                          ((4096, 11008), 50, 3), ((1000, 1024), 70, 17), ((4096, 4096), 70, 33)])
def test_noalloc_matches_sp_linear_on_two_calls_in_a_row(oracle, shape, pct, M):
    import torch

    from paper_2405_03594_gb300 import sp

    N, K = shape
    g = np.random.default_rng(N + K + M)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    x = synth.activations(M, K, g)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    xd = gu.bf16_to_dev(x)
    ref = gu.bf16_from_dev(h.linear(xd, path="cuda_core"))  # the existing entry point
    outs = []
    for _ in range(2):
        y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
        h.linear_noalloc(xd, y)
        sp.check()
        outs.append(gu.bf16_from_dev(y))
    exact = oracle.linear_bf16(x, W, mask)
    for y in outs:
        gu.assert_close(y, ref, f"noalloc {N}x{K} M={M}")
        gu.assert_close(y, exact, f"noalloc {N}x{K} M={M} vs the oracle")
