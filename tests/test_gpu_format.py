"""GPU compress / decompress against the oracle: bit-exact bytes, offsets and round trip."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu
from tests.test_oracle import _golden_2x8

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2405_03594_gb300 import sp as _sp

    return _sp


SHAPES = [(1, 8), (2, 64), (130, 72), (300, 200), (257, 136), (128, 1024), (1000, 4096), (129, 11008)]


def _compress_dev(sp, W, mask, int8):
    if int8:
        q, s = synth.quantize_int8(W, mask)
        return q, s, sp.compress(gu.i8_to_dev(q), gu.u8_to_dev(mask), gu.f32_to_dev(s))
    return W, None, sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))


@pytest.mark.parametrize("N,K", SHAPES)
@pytest.mark.parametrize("pct", [0, 50, 70, 100])
@pytest.mark.parametrize("int8", [False, True])
def test_compress_bytes_and_roundtrip(sp, oracle, N, K, pct, int8):
    g = np.random.default_rng(N * 31 + K + pct)
    W = synth.weight(N, K, g)
    mask = synth.magnitude_mask(W, pct)
    vals, s, h = _compress_dev(sp, W, mask, int8)
    buf, off = h.copy_out()
    obuf, ooff = oracle.compress(vals, mask)
    assert np.array_equal(off, ooff)
    assert np.array_equal(buf, obuf)
    assert int(h.info.nnz) == int(mask.sum()) and int(h.info.bytes) == obuf.size
    back = h.decompress()
    import torch

    torch.cuda.synchronize()
    if int8:
        got = back.cpu().numpy()
        expect = np.where(mask != 0, vals, 0).astype(np.int8)
        assert np.array_equal(got, expect)
    else:
        got = gu.bf16_bits_from_dev(back)
        assert np.array_equal(got, np.where(mask != 0, W, 0).astype(np.uint16))
    sp.check()


def test_hand_derived_example_on_gpu(sp, oracle):
    g, N, K, W, mask = _golden_2x8()
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    buf, off = h.copy_out()
    total = int(g["expect_total_bytes"][0])
    assert list(off) == [0, total]
    assert list(buf[:1024].view(np.uint64)[:2]) == [int(v, 16) for v in g["expect_mask_u64"]]
    vb = [int(v, 16) for v in g["expect_value_bytes"]]
    assert list(buf[1024:1024 + len(vb)]) == vb and not buf[1024 + len(vb):].any()


def test_negative_zero_and_kept_zero(sp, oracle):
    N, K = 3, 16
    W = np.zeros((N, K), dtype=np.uint16)
    W[0, 3] = 0x8000
    W[1, 5] = 0x3F80
    mask = np.zeros((N, K), dtype=np.uint8)
    mask[0, 3] = 1
    mask[2, 7] = 1
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    buf, _ = h.copy_out()
    assert list(buf[1024:1028].view(np.uint16)) == [0x8000, 0x0000]
    back = gu.bf16_bits_from_dev(h.decompress())
    assert back[0, 3] == 0x8000 and back[1, 5] == 0


@pytest.mark.parametrize("name", list(synth.LLAMA2_7B_SHAPES))
def test_full_size_llama_shapes_70pct(sp, oracle, name):
    N, K = synth.LLAMA2_7B_SHAPES[name]
    W, mask, _ = synth.layer_inputs(name, 70, 1)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    buf, off = h.copy_out()
    obuf, ooff = oracle.compress(W, mask)
    assert np.array_equal(off, ooff) and np.array_equal(buf, obuf)
    per_row = {4096: 1229, 11008: 3302}[K]
    assert int(h.info.nnz) == N * per_row


def test_clone_has_identical_bytes(sp):
    g = np.random.default_rng(1)
    W = synth.weight(300, 200, g)
    mask = synth.magnitude_mask(W, 50)
    h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
    c = h.clone()
    a, ao = h.copy_out()
    b, bo = c.copy_out()
    assert np.array_equal(a, b) and np.array_equal(ao, bo)
