"""The linear-stack decode step (INT8 weights, 70%): every sparse linear (with its fused
residual or gate * up epilogue where the batch runs on the CUDA cores) is checked against the
float64 oracle on the GPU's own inputs, the glue against the oracle's glue, and a CUDA-graph
replay against the eager step."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stack():
    import torch

    from paper_2405_03594_gb300.stack import LinearStack

    torch.cuda.set_device(0)
    return LinearStack(layers=2, pct=70, int8=True, max_m=64)


def _bits(t):
    return gu.bf16_bits_from_dev(t)


@pytest.mark.parametrize("M", [1, 4, 64])
def test_each_linear_matches_oracle_on_gpu_inputs(stack, oracle, M):
    x = synth.activations(M, 4096, synth.rng(0, 7, 0, synth.STREAM_X))
    stack.h[:M].copy_(gu.bf16_to_dev(x))
    rec = []
    stack.step(M, record=rec)
    from paper_2405_03594_gb300 import sp

    sp.check()
    assert len(rec) == 4 * stack.layers
    rows_rng = np.random.default_rng(M)
    for item in rec:
        layer, name = item[0], item[1]
        N = stack.host_of(layer, name)[0].shape[0]
        rows = None if M <= 4 else np.sort(rows_rng.choice(N, 256, replace=False))
        pairs = None if M <= 4 else np.sort(rows_rng.choice(N // 2, 128, replace=False))
        gu.check_stack_record(oracle, stack, item, rows=rows, sample_pairs=pairs, what=f"layer {layer} {name} M={M}")
    # batches on the CUDA-core kernels fold the glue into the linears' epilogues
    assert {e[4] for e in rec} == ({"store", "residual", "pair_product"} if stack.fuses(M) else {"store"})


def test_glue_matches_oracle(stack, oracle):
    import torch

    from paper_2405_03594_gb300 import sp

    M = 5
    g = np.random.default_rng(3)
    h = synth.activations(M, 4096, g)
    a = synth.activations(M, 4096, g)
    r = synth.activations(1, 4096, g)[0]
    hd = gu.bf16_to_dev(h)
    sp.residual_add(hd, gu.bf16_to_dev(a), gu.bf16_to_dev(r))
    ref = oracle.residual_add(h, a, r)
    got = gu.bf16_from_dev(hd)
    # FP32 arithmetic with one bf16 rounding: within one bf16 ulp of the float64 value
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0**-7 + 1e-30)
    gg = synth.activations(M, 2 * 11008, g)
    out = torch.empty((M, 11008), dtype=torch.bfloat16, device="cuda")
    sp.mul_halves(out, gu.bf16_to_dev(gg))
    ref = oracle.mul_halves(gg)
    got = gu.bf16_from_dev(out)
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0**-8 + 1e-30)
    src = gu.bf16_to_dev(synth.activations(M, 12288, g))
    dst = torch.empty((M, 4096), dtype=torch.bfloat16, device="cuda")
    sp.copy_columns(dst, src, 8192)
    assert np.array_equal(_bits(dst), _bits(src)[:, 8192:])
    sp.check()


@pytest.mark.parametrize("M", [1, 16])
def test_graph_replay_equals_eager_step(stack, M):
    import torch

    x = gu.bf16_to_dev(synth.activations(M, 4096, synth.rng(0, 8, 0, synth.STREAM_X)))
    stack.set_input(x)
    stack.step(M)
    eager = _bits(stack.h[:M]).copy()
    assert np.isfinite(synth.bf16_to_f32(eager)).all()
    g = stack.capture(M)
    for _ in range(3):  # every replay restarts from the saved input
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(_bits(stack.h[:M]), eager)
