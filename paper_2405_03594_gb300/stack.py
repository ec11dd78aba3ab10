"""Decode step of a Llama-2-7B linear-only stack on libsp.

Per layer, four sparse linears and the elementwise glue of include/sp_stack.h:

    qkv = x.Wqkv^T            [M, 12288]      (sparse linear)
    v   = qkv[:, 8192:12288]                   (read in place at M = 1, else sp_copy_columns)
    h   = h + v.Wo^T + r_l                      (sparse linear + residual)
    a   = gate(h) * up(h)     [M, 11008]      (sparse linear + gate * up)
    h   = h + a.Wdown^T + r'_l                  (sparse linear + residual)

By default (`fused`) the gate/up weight holds interleaved rows (gate_j, up_j), and where a
batch runs on the CUDA-core decode kernels the residual adds and the gate * up product are
those kernels' output epilogues (sp_linear_epi): four launches per layer.  Tensor-core
batches, and stacks built with fused=False, run each linear into a buffer and the glue as
its own launch (sp_residual_add; sp_mul_pairs on interleaved rows, sp_mul_halves on the
[gate, up] layout).  All arithmetic runs in libsp kernels; PyTorch only holds the buffers.  The layers are
device copies of one seeded layer (each its own HBM buffers, so a step streams the full
32-layer weight set), or each layer's own seeded inputs (`host_layers`: distinct weights,
or a per-layer sparsity profile).  `capture()` records one step as a single CUDA graph.

`ChainStack` runs the same step (for batches of up to 4 rows) as one persistent launch of
sp_chain_run: the glue is fused into the linears' epilogues (v is read in place from
qkv; h + o(v) + r and h + down(a) + r' are residual epilogues), and the gate/up weight is
stored with its rows interleaved (gate_j, up_j) so that the gate*up product is the pair
epilogue of one row block.
"""
from __future__ import annotations

import numpy as np
import torch

from . import sp, synth

SHAPES = ("qkv", "o", "gate_up", "down")
D_MODEL = 4096
D_FF = 11008
# Initial weight scale of the stack: with N(0, 0.02^2) weights, 70% magnitude masks and
# no normalisation, the gate*up product makes activations overflow within a few layers;
# N(0, 0.003^2) keeps them O(10) through 32 layers.
STACK_WEIGHT_STD = 0.003


def host_layer(pct, int8: bool, seed: int = 0, std: float = STACK_WEIGHT_STD, layer: int = 0):
    """Seeded host inputs of one layer: {shape: (values, mask, scale or None)}."""
    return synth.stack_layer(pct, int8, seed=seed, layer=layer, std=std)


def _compress_layer(host: dict, dev, interleave_gate_up: bool = False) -> dict:
    """{shape: SparseMatrix} of one layer's host inputs (gate/up rows interleaved for the
    chained step's pair epilogue)."""
    out = {}
    for name in SHAPES:
        vals, mask, s = host[name]
        if interleave_gate_up and name == "gate_up":
            vals, mask = interleave_rows(vals, D_FF), interleave_rows(mask, D_FF)
            s = None if s is None else interleave_rows(s, D_FF)
        vals, mask = np.ascontiguousarray(vals), np.ascontiguousarray(mask)
        if s is not None:
            out[name] = sp.compress(torch.from_numpy(vals).to(dev), torch.from_numpy(mask).to(dev),
                                    torch.from_numpy(np.ascontiguousarray(s)).to(dev))
        else:
            out[name] = sp.compress(torch.from_numpy(vals.view(np.int16)).to(dev).view(torch.bfloat16),
                                    torch.from_numpy(mask).to(dev))
    return out


def _layer_mats(layers: int, host, host_layers, dev, interleave_gate_up: bool) -> dict:
    """{shape: [SparseMatrix per layer]}: device copies of one layer (host), or each layer's
    own inputs (host_layers, one dict per layer)."""
    if host_layers is not None:
        per = [_compress_layer(hl, dev, interleave_gate_up) for hl in host_layers]
        return {name: [p[name] for p in per] for name in SHAPES}
    one = _compress_layer(host, dev, interleave_gate_up)
    return {name: [one[name]] + [one[name].clone() for _ in range(layers - 1)] for name in SHAPES}


def _must(ran: bool):
    if not ran:  # fuses() chose the epilogue path for a batch that the library runs on tensor cores
        raise RuntimeError("sp_linear_epi declined a batch the stack expected to fuse")


class LinearStack:
    """host: one layer's inputs, copied to every layer; host_layers: each layer's own inputs
    (then `layers` is their count).  fused (automatic path only): the gate/up weight holds
    interleaved rows and, for batches that run on the CUDA-core kernels, the residual adds and
    the gate * up product are the linears' epilogues (sp_linear_epi); tensor-core batches keep
    the separate glue launches (sp_residual_add, sp_mul_pairs)."""

    def __init__(self, layers: int = 32, pct: int = 70, int8: bool = True, max_m: int = 64, seed: int = 0,
                 device=None, host=None, path: str = "auto", host_layers=None, fused: bool = True):
        self.dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
        if host_layers is not None:
            layers = len(host_layers)
        self.layers, self.max_m, self.path = layers, max_m, path
        self.fused = fused and path == "auto"
        self.host = None if host_layers is not None else (host_layer(pct, int8, seed) if host is None else host)
        self.host_layers = host_layers
        self.mats = _layer_mats(layers, self.host, host_layers, self.dev, self.fused)
        g = synth.rng(seed, 0, 9, synth.STREAM_RESID)
        r = synth.activations(2 * layers, D_MODEL, g)
        rt = torch.from_numpy(r.view(np.int16)).to(self.dev).view(torch.bfloat16)
        self.r1 = [rt[2 * l].contiguous() for l in range(layers)]
        self.r2 = [rt[2 * l + 1].contiguous() for l in range(layers)]
        bf = dict(dtype=torch.bfloat16, device=self.dev)
        self.h = torch.zeros((max_m, D_MODEL), **bf)
        self.x0 = torch.zeros((max_m, D_MODEL), **bf)  # the step's input token embeddings
        self.qkv = torch.empty((max_m, 3 * D_MODEL), **bf)
        self.v = torch.empty((max_m, D_MODEL), **bf)
        self.o = torch.empty((max_m, D_MODEL), **bf)
        self.gu = torch.empty((max_m, 2 * D_FF), **bf)
        self.a = torch.empty((max_m, D_FF), **bf)
        self.d = torch.empty((max_m, D_MODEL), **bf)
        ws = max(self.mats[n][0].workspace_size(max_m) for n in SHAPES)
        self.ws = torch.zeros(max(ws, 256), dtype=torch.uint8, device=self.dev)
        torch.cuda.synchronize()

    def weight_bytes(self) -> int:
        return sum(int(m.info.bytes) + int(m.info.scale_bytes) for n in SHAPES for m in self.mats[n])

    def host_of(self, layer: int, name: str):
        """Host (values, mask, scale) of `name` in `layer` (gate/up with interleaved rows when
        fused)."""
        vals, mask, s = (self.host_layers[layer] if self.host_layers is not None else self.host)[name]
        if self.fused and name == "gate_up":
            vals, mask = interleave_rows(vals, D_FF), interleave_rows(mask, D_FF)
            s = None if s is None else interleave_rows(s, D_FF)
        return vals, mask, s

    def fuses(self, M: int) -> bool:
        """Whether a step of M rows folds the residual adds and gate * up into the linears."""
        return self.fused and all(self.mats[n][0].kernel_name(M) != "linear_tc_kernel" for n in SHAPES)

    def launches_per_step(self, M: int, reset: bool = True) -> int:
        """libsp kernels per step: the four sparse linears (as many launches as the library
        reports for M rows) and the glue kernels per layer: the v-block copy (none at M = 1,
        where the o linear reads it in place), and the two residual adds and gate * up unless
        they are the linears' epilogues; plus the input copy."""
        per_layer = sum(self.mats[n][0].launch_count(M, self.path) for n in SHAPES)
        glue = (0 if M == 1 else 1) + (0 if self.fuses(M) else 3)
        return self.layers * (per_layer + glue) + (1 if reset else 0)

    def set_input(self, x: torch.Tensor):
        """Token embeddings [M, 4096] bf16 for the next steps."""
        M = x.shape[0]
        self.x0[:M].copy_(x)
        self.h[:M].copy_(x)

    def step(self, M: int, record=None, stream=None, reset: bool = False):
        """One decode step for the first M rows of self.h (in place); with reset=True it
        starts from the saved input (set_input).  If `record` is a list, each linear appends
        (layer, shape, input, output, epilogue, h before the linear) copies: epilogue "store"
        (output = the linear's result), "residual" (output = h after it, in place) or
        "pair_product" (output = gate * up)."""
        kw = dict(workspace=self.ws, path=self.path, stream=stream)
        h, qkv, v, o, gu, a, d = (t[:M] for t in (self.h, self.qkv, self.v, self.o, self.gu, self.a, self.d))
        fuse = self.fuses(M)
        if reset:
            sp.copy_columns(h, self.x0[:M], 0, stream=stream)
        for l in range(self.layers):
            self.mats["qkv"][l].linear(h, out=qkv, **kw)
            if record is not None:
                record.append((l, "qkv", h.clone(), qkv.clone(), "store", None))
            # one row of qkv's v block is already a contiguous, 16-byte aligned vector: the o
            # linear reads it in place; more rows are gathered by one glue launch
            vin = qkv[:, 2 * D_MODEL:] if M == 1 else v
            if M != 1:
                sp.copy_columns(v, qkv, 2 * D_MODEL, stream=stream)
            self._residual("o", l, vin, o, h, self.r1[l], fuse, record, stream)
            if fuse:
                hb = h.clone() if record is not None else None
                _must(self.mats["gate_up"][l].linear_epi(h, a, "pair_product", workspace=self.ws, stream=stream))
                if record is not None:
                    record.append((l, "gate_up", hb, a.clone(), "pair_product", None))
            else:
                self.mats["gate_up"][l].linear(h, out=gu, **kw)
                if record is not None:
                    record.append((l, "gate_up", h.clone(), gu.clone(), "store", None))
                (sp.mul_pairs if self.fused else sp.mul_halves)(a, gu, stream=stream)
            self._residual("down", l, a, d, h, self.r2[l], fuse, record, stream)

    def _residual(self, name, l, x, tmp, h, r, fuse, record, stream):
        """h <- bf16((h + bf16(linear(x))) + r): the linear's epilogue, or a linear into tmp
        and the glue add."""
        hb = h.clone() if record is not None else None
        if fuse:
            _must(self.mats[name][l].linear_epi(x, h, "residual", r, workspace=self.ws, stream=stream))
            if record is not None:
                record.append((l, name, x.clone(), h.clone(), "residual", hb))
            return
        self.mats[name][l].linear(x, out=tmp, workspace=self.ws, path=self.path, stream=stream)
        if record is not None:
            record.append((l, name, x.clone(), tmp.clone(), "store", hb))
        sp.residual_add(h, tmp, r, stream=stream)

    def capture(self, M: int) -> torch.cuda.CUDAGraph:
        """One decode step from the saved input, recorded as a single CUDA graph."""
        self.step(M, reset=True)  # warm: per-device kernel attributes are set outside the capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step(M, reset=True)
        torch.cuda.synchronize()
        return g


def interleave_rows(a: np.ndarray, half: int) -> np.ndarray:
    """Rows [r_0, ..., r_{F-1}, r_F, ..., r_{2F-1}] -> [r_0, r_F, r_1, r_{F+1}, ...]."""
    out = np.empty_like(a)
    out[0::2] = a[:half]
    out[1::2] = a[half:]
    return out


class ChainStack:
    """The 32-layer linear stack as one sp_chain_run call per decode step (m <= 4 rows)."""

    def __init__(self, layers: int = 32, pct: int = 70, int8: bool = False, max_m: int = 4, seed: int = 0,
                 device=None, host=None, host_layers=None):
        self.dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
        if host_layers is not None:
            layers = len(host_layers)
        self.layers, self.max_m = layers, max_m
        self.host = None if host_layers is not None else (host_layer(pct, int8, seed) if host is None else host)
        self.host_layers = host_layers
        self.mats = _layer_mats(layers, self.host, host_layers, self.dev, True)
        g = synth.rng(seed, 0, 9, synth.STREAM_RESID)
        r = synth.activations(2 * layers, D_MODEL, g)
        rt = torch.from_numpy(r.view(np.int16)).to(self.dev).view(torch.bfloat16)
        self.r1 = [rt[2 * l].contiguous() for l in range(layers)]
        self.r2 = [rt[2 * l + 1].contiguous() for l in range(layers)]
        bf = dict(dtype=torch.bfloat16, device=self.dev)
        self.h = torch.zeros((max_m, D_MODEL), **bf)
        self.x0 = torch.zeros((max_m, D_MODEL), **bf)
        self.qkv = torch.empty((max_m, 3 * D_MODEL), **bf)
        self.a = torch.empty((max_m, D_FF), **bf)
        self._chains = {}
        torch.cuda.synchronize()

    def weight_bytes(self) -> int:
        return sum(int(m.info.bytes) + int(m.info.scale_bytes) for n in SHAPES for m in self.mats[n])

    def host_of(self, layer: int, name: str):
        """Host (values, mask, scale) of `name` in `layer`, in the stored row order (gate/up
        interleaved)."""
        vals, mask, s = (self.host_layers[layer] if self.host_layers is not None else self.host)[name]
        if name == "gate_up":
            vals, mask = interleave_rows(vals, D_FF), interleave_rows(mask, D_FF)
            s = None if s is None else interleave_rows(s, D_FF)
        return vals, mask, s

    def ops(self, M: int):
        """The chain of one decode step: four linears per layer."""
        h, qkv, a = self.h[:M], self.qkv[:M], self.a[:M]
        v = qkv[:, 2 * D_MODEL:]
        out = []
        for l in range(self.layers):
            out.append((self.mats["qkv"][l], h, qkv, "store", None))
            out.append((self.mats["o"][l], v, h, "residual", self.r1[l]))
            out.append((self.mats["gate_up"][l], h, a, "pair_product", None))
            out.append((self.mats["down"][l], a, h, "residual", self.r2[l]))
        return out

    def chain(self, M: int) -> "sp.Chain":
        if M not in self._chains:
            self._chains[M] = sp.Chain(self.ops(M), M)
        return self._chains[M]

    def set_input(self, x: torch.Tensor):
        M = x.shape[0]
        self.x0[:M].copy_(x)
        self.h[:M].copy_(x)

    def step(self, M: int, stream=None, reset: bool = True):
        """One decode step for the first M rows of self.h (in place): two library launches
        (the copy of the saved input when reset=True, then the whole chain)."""
        c = self.chain(M)
        if reset:
            sp.copy_columns(self.h[:M], self.x0[:M], 0, stream=stream)
        c.run(stream=stream)

    def launches_per_step(self, M: int, reset: bool = True) -> int:
        return (4 * self.layers + 159) // 160 + (1 if reset else 0)
