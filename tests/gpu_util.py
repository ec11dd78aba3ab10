"""Helpers for the GPU parity tests: host <-> device marshalling and the acceptance
tolerances (max |err| <= 1e-2 * max|ref| and relative Frobenius error <= 5e-3
against the float64 oracle)."""
import numpy as np

from paper_2405_03594_gb300 import synth

MAX_REL = 1e-2
FRO_REL = 5e-3


def dev():
    import torch

    return torch.device("cuda", 0)


def bf16_to_dev(a_u16):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a_u16).view(np.int16)).to(dev()).view(torch.bfloat16)


def u8_to_dev(a):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint8)).to(dev())


def i8_to_dev(a):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int8)).to(dev())


def f32_to_dev(a):
    import torch

    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev())


def bf16_bits_from_dev(t):
    import torch

    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def bf16_from_dev(t):
    return synth.bf16_to_f32(bf16_bits_from_dev(t)).astype(np.float64)


def errors(y, ref):
    scale = np.abs(ref).max()
    maxerr = np.abs(y - ref).max() if y.size else 0.0
    nref = np.linalg.norm(ref)
    fro = np.linalg.norm(y - ref) / nref if nref > 0 else np.linalg.norm(y - ref)
    return maxerr, scale, fro


def assert_close(y, ref, what=""):
    maxerr, scale, fro = errors(y, ref)
    assert maxerr <= MAX_REL * scale + 1e-30 and fro <= FRO_REL, (
        f"{what}: max|err|={maxerr:.3e} (limit {MAX_REL * scale:.3e}), rel_fro={fro:.3e} (limit {FRO_REL})")
    return maxerr / scale if scale else 0.0, fro


def check_stack_record(oracle, st, item, rows=None, sample_pairs=None, what=""):
    """One recorded linear of a LinearStack step, (layer, shape, input, output, epilogue, h
    before), against the float64 oracle on the GPU's own inputs: store -> the linear;
    residual -> h before + the linear + r; pair product -> the gate and up outputs' product
    (rows 2j, 2j + 1 of the interleaved weight).  rows / sample_pairs: output rows / pairs to
    check (all by default)."""
    import numpy as np

    from paper_2405_03594_gb300 import synth

    layer, name, inp, out, epi, prev = item
    vals, mask, s = st.host_of(layer, name)
    x = bf16_bits_from_dev(inp)
    y = bf16_from_dev(out)
    assert np.isfinite(y).all()

    def lin(rr):
        v, m = vals[rr], mask[rr]
        if s is not None:
            return oracle.linear_int8(x, v, m, s[rr])
        return oracle.linear_bf16(x, v, m)

    N = vals.shape[0]
    if epi == "pair_product":
        j = np.arange(N // 2) if sample_pairs is None else sample_pairs
        rr = np.stack([2 * j, 2 * j + 1], axis=1).reshape(-1)
        yl = lin(rr)
        assert_close(y[:, j], yl[:, 0::2] * yl[:, 1::2], what)
        return
    rr = np.arange(N) if rows is None else rows
    ref = lin(rr)
    if epi == "residual":
        r = synth.bf16_to_f32(bf16_bits_from_dev(st.r1[layer] if name == "o" else st.r2[layer])).astype(np.float64)
        ref = bf16_from_dev(prev)[:, rr].astype(np.float64) + ref + r[rr]
    assert_close(y[:, rr], ref, what)
