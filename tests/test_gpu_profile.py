"""Linear stacks whose layers differ: every layer its own seeded weights (the INT8 stack of
32 distinct layers, M = 1), and a per-layer sparsity profile (60 .. 80 %, mean 70 %; the
stand-in for an outlier-weighted layerwise profile).  Every linear is checked against the
float64 oracle on the GPU's own inputs, through both the graph-of-launches stack and the
one-launch chained step."""
import multiprocessing as mp
import os

import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

STACK_STD = 0.003  # the stack's weight scale (paper_2405_03594_gb300.stack.STACK_WEIGHT_STD)


def _gen_layer(args):
    """(pct or {shape: pct}, int8, layer) -> one layer's host inputs; runs in a worker."""
    pct, int8, layer = args
    return synth.stack_layer(pct, int8, seed=0, layer=layer, std=STACK_STD)


def _gen_layers(specs):
    """Host inputs of several layers, generated in parallel (spawned workers: no CUDA state)."""
    n = max(1, min(len(specs), os.cpu_count() or 1, 16))
    with mp.get_context("spawn").Pool(n) as pool:
        return pool.map(_gen_layer, specs)


def _lin(oracle, host, x_bits, rows=None):
    vals, mask, s = host
    if rows is not None:
        vals, mask = vals[rows], mask[rows]
        s = None if s is None else s[rows]
    return oracle.linear_int8(x_bits, vals, mask, s) if s is not None else oracle.linear_bf16(x_bits, vals, mask)


def _check_recorded(oracle, st, rec, M, sample=None, seed=0):
    g = np.random.default_rng(seed)
    for item in rec:
        layer, name = item[0], item[1]
        N = st.host_of(layer, name)[0].shape[0]
        rows = None if sample is None else np.sort(g.choice(N, sample, replace=False))
        pairs = None if sample is None else np.sort(g.choice(N // 2, sample // 2, replace=False))
        gu.check_stack_record(oracle, st, item, rows=rows, sample_pairs=pairs, what=f"layer {layer} {name} M={M}")


def test_int8_stack_32_distinct_layers_m1(oracle):
    """The 32-layer INT8 stack at 70 % with distinct seeded weights in every layer, one decode
    step at M = 1: all 128 linears, every output row, on the inputs the GPU produced."""
    import torch

    from paper_2405_03594_gb300 import sp
    from paper_2405_03594_gb300.stack import LinearStack

    torch.cuda.set_device(0)
    hosts = _gen_layers([(70, True, l) for l in range(32)])
    st = LinearStack(int8=True, max_m=1, host_layers=hosts)
    assert st.layers == 32
    # distinct layers: the first linear's compressed bytes differ between layers 0 and 1
    assert not np.array_equal(st.mats["qkv"][0].copy_out()[0], st.mats["qkv"][1].copy_out()[0])
    x = synth.activations(1, 4096, synth.rng(0, 7, 0, synth.STREAM_X))
    st.h[:1].copy_(gu.bf16_to_dev(x))
    rec = []
    st.step(1, record=rec)
    sp.check()
    assert len(rec) == 128
    _check_recorded(oracle, st, rec, 1)


@pytest.fixture(scope="module")
def profile_hosts():
    """Eight bf16 layers at the seeded per-layer sparsity profile (mean 70 %)."""
    prof = synth.layer_sparsity_profile(8)
    assert sum(prof) == 70 * 8 and min(prof) == 60 and max(prof) == 80
    return prof, _gen_layers([(p, False, l) for l, p in enumerate(prof)])


@pytest.mark.parametrize("M", [1, 4])
def test_profile_linear_stack_each_linear(oracle, profile_hosts, M):
    from paper_2405_03594_gb300 import sp
    from paper_2405_03594_gb300.stack import LinearStack

    prof, hosts = profile_hosts
    st = LinearStack(int8=False, max_m=4, host_layers=hosts)
    for l, p in enumerate(prof):  # each layer at its own sparsity
        N, K = synth.LLAMA2_7B_SHAPES["gate_up"]
        assert int(st.mats["gate_up"][l].info.nnz) == N * (K - synth.n_pruned(p, K))
    x = synth.activations(M, 4096, synth.rng(0, 8, 0, synth.STREAM_X))
    st.h[:M].copy_(gu.bf16_to_dev(x))
    rec = []
    st.step(M, record=rec)
    sp.check()
    _check_recorded(oracle, st, rec, M, sample=512, seed=M)


def test_profile_chain_stack_each_linear(oracle, profile_hosts):
    """The same layers as one chained launch: the chain cut to k linears leaves the state from
    which linear k is checked (the chain is deterministic)."""
    from paper_2405_03594_gb300 import sp
    from paper_2405_03594_gb300.stack import D_MODEL, ChainStack

    prof, hosts = profile_hosts
    M = 2
    cs = ChainStack(int8=False, max_m=4, host_layers=hosts)
    x0 = synth.activations(M, D_MODEL, synth.rng(0, 9, 0, synth.STREAM_X))
    ops = cs.ops(M)
    names = ["qkv", "o", "gate_up", "down"]
    r_host = [gu.bf16_bits_from_dev(r) for pair in zip(cs.r1, cs.r2) for r in pair]
    g = np.random.default_rng(3)

    def state(k):
        cs.h[:M].copy_(gu.bf16_to_dev(x0))
        cs.qkv.fill_(float("nan"))
        cs.a.fill_(float("nan"))
        if k:
            sp.Chain(ops[:k], M).run()
        sp.check()
        f = gu.bf16_bits_from_dev
        return {"h": f(cs.h[:M]).copy(), "qkv": f(cs.qkv[:M]).copy(), "a": f(cs.a[:M]).copy()}

    prev = state(0)
    for k in range(1, len(ops) + 1):
        cur = state(k)
        l, name = (k - 1) // 4, names[(k - 1) % 4]
        host = cs.host_of(l, name)
        what = f"chained linear {k - 1} ({name}, layer {l}, {prof[l]}%)"
        f64 = lambda b: synth.bf16_to_f32(b).astype(np.float64)  # noqa: E731
        if name == "qkv":
            rows = np.sort(g.choice(host[0].shape[0], 384, replace=False))
            gu.assert_close(f64(cur["qkv"])[:, rows], _lin(oracle, host, prev["h"], rows), what)
        elif name in ("o", "down"):
            xin = prev["qkv"][:, 2 * D_MODEL:] if name == "o" else prev["a"]
            rows = np.sort(g.choice(host[0].shape[0], 384, replace=False))
            r = f64(r_host[2 * l + (0 if name == "o" else 1)])
            ref = f64(prev["h"])[:, rows] + _lin(oracle, host, np.ascontiguousarray(xin), rows) + r[rows]
            gu.assert_close(f64(cur["h"])[:, rows], ref, what)
        else:
            j = np.sort(g.choice(host[0].shape[0] // 2, 384, replace=False))
            rows = np.stack([2 * j, 2 * j + 1], axis=1).reshape(-1)
            y = _lin(oracle, host, prev["h"], rows)
            gu.assert_close(f64(cur["a"])[:, j], y[:, 0::2] * y[:, 1::2], what)
        prev = cur
