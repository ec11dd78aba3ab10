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
