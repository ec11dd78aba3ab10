"""sp_linear_epi (a sparse linear with the stack's glue as its output epilogue) and the
interleaved gate * up glue sp_mul_pairs, on the GPU: the fused results equal sp_linear
followed by the glue call bit for bit (same kernel, same roundings), and match the float64
oracle; batches that would run on the tensor-core kernel are declined without a launch."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2405_03594_gb300 import sp as _sp

    return _sp


def _matrix(sp, N, K, pct, int8, seed):
    g = np.random.default_rng(seed)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    if int8:
        q, s = synth.quantize_int8(W, mask)
        return (q, mask, s), sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    return (W, mask, None), sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))


def _lin(oracle, host, x):
    v, m, s = host
    return oracle.linear_int8(x, v, m, s) if s is not None else oracle.linear_bf16(x, v, m)


# (N, K): ragged tiles, a Llama o shape (cluster split at M = 1), a matrix of 320 row blocks
# (more than two per SM slot: stream-K), and gate/up (pairs)
SHAPES = [(300, 200), (4096, 4096), (40960, 256), (22016, 4096)]
CASES = [(False, 1), (False, 3), (False, 4), (False, 5), (False, 10), (True, 1), (True, 4), (True, 13)]


@pytest.mark.parametrize("N,K", SHAPES)
@pytest.mark.parametrize("int8,M", CASES)
def test_epilogues_equal_linear_plus_glue_and_oracle(sp, oracle, N, K, int8, M):
    import torch

    host, h = _matrix(sp, N, K, 70, int8, N + K + M)
    g = np.random.default_rng(M)
    x = synth.activations(M, K, g)
    h0 = synth.activations(M, N, g)
    r = synth.activations(1, N, g)[0]
    xd, rd = gu.bf16_to_dev(x), gu.bf16_to_dev(r)
    ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device="cuda")
    y = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    h.linear(xd, out=y, workspace=ws)
    ref = _lin(oracle, host, x)

    # store
    ys = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    assert h.linear_epi(xd, ys, "store", workspace=ws)
    assert np.array_equal(gu.bf16_bits_from_dev(ys), gu.bf16_bits_from_dev(y))

    # residual, in place
    hf = gu.bf16_to_dev(h0)
    assert h.linear_epi(xd, hf, "residual", rd, workspace=ws)
    if N % 8 == 0:  # the glue call's vector width
        hg = gu.bf16_to_dev(h0)
        sp.residual_add(hg, y, rd)
        assert np.array_equal(gu.bf16_bits_from_dev(hf), gu.bf16_bits_from_dev(hg))
    want = synth.bf16_to_f32(h0).astype(np.float64) + ref + synth.bf16_to_f32(r).astype(np.float64)
    gu.assert_close(gu.bf16_from_dev(hf), want, f"residual {N}x{K} M={M}")

    # pair product of rows (2j, 2j + 1)
    a = torch.full((M, N // 2), float("nan"), dtype=torch.bfloat16, device="cuda")
    assert h.linear_epi(xd, a, "pair_product", workspace=ws)
    b = torch.empty((M, N // 2), dtype=torch.bfloat16, device="cuda")
    if (N // 2) % 8 == 0:
        sp.mul_pairs(b, y)
        assert np.array_equal(gu.bf16_bits_from_dev(a), gu.bf16_bits_from_dev(b))
    gu.assert_close(gu.bf16_from_dev(a), ref[:, 0::2] * ref[:, 1::2], f"pair product {N}x{K} M={M}")
    sp.check()


def test_tensor_core_batches_are_declined(sp):
    import torch

    _, h = _matrix(sp, 4096, 4096, 70, False, 1)
    M = 64
    x = gu.bf16_to_dev(synth.activations(M, 4096, np.random.default_rng(0)))
    ws = torch.zeros(max(h.workspace_size(M), 256), dtype=torch.uint8, device="cuda")
    assert h.kernel_name(M) == "linear_tc_kernel"
    y = torch.full((M, 4096), 7.0, dtype=torch.bfloat16, device="cuda")
    assert not h.linear_epi(x, y, "store", workspace=ws)
    torch.cuda.synchronize()
    assert bool((y == 7.0).all())  # nothing launched
    sp.check()


def test_argument_errors(sp):
    import ctypes

    import torch

    _, h = _matrix(sp, 301, 64, 50, False, 2)  # odd N
    x = torch.zeros((1, 64), dtype=torch.bfloat16, device="cuda")
    y = torch.zeros((1, 301), dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(max(h.workspace_size(1), 256), dtype=torch.uint8, device="cuda")
    lib = sp._lib
    call = lambda epi, r: lib.sp_linear_epi(h.handle, x.data_ptr(), 1, y.data_ptr(), epi, r, ws.data_ptr(),
                                            ws.numel(), None)
    assert call(2, None) == 1  # pair product with an odd N
    assert call(1, None) == 1  # residual without r
    assert call(7, None) == 1  # unknown epilogue
    assert call(0, None) == 0  # store
    assert lib.sp_linear_epi(None, x.data_ptr(), 1, y.data_ptr(), 0, None, ws.data_ptr(), ws.numel(), None) == 7
    assert lib.sp_linear_epi(h.handle, x.data_ptr(), 1, y.data_ptr(), 0, None, None, 0, None) == 8
    assert lib.sp_mul_pairs(ctypes.c_void_p(y.data_ptr()), ctypes.c_void_p(x.data_ptr()), 1, 12, None) == 2
    sp.check()


@pytest.mark.parametrize("M,F", [(1, 11008), (5, 64), (16, 4096)])
def test_mul_pairs_matches_oracle(sp, oracle, M, F):
    import torch

    g = synth.activations(M, 2 * F, np.random.default_rng(F + M))
    out = torch.empty((M, F), dtype=torch.bfloat16, device="cuda")
    sp.mul_pairs(out, gu.bf16_to_dev(g))
    ref = oracle.mul_halves(np.concatenate([g[:, 0::2], g[:, 1::2]], axis=1))
    got = gu.bf16_from_dev(out)
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0**-8 + 1e-30)
    sp.check()
