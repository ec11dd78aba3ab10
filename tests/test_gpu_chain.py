"""sp_chain_run: a chain of sparse linears in one persistent launch (the decode step of a
linear stack) against the float64 oracle.

Every linear of a chain is checked on the GPU's own inputs: the chain is deterministic,
so the state after its first k linears is the final state of the chain cut to k linears,
and linear k is checked from that state (store: y = x.W^T; residual: y_new = y_old +
x.W^T + r; pair product: y[:, j] = (x.W^T)[:, 2j] * (x.W^T)[:, 2j+1]).  Buffers that a
linear reads before anything wrote them start as NaN, so a linear that read its input too
early fails.  Tolerances are the acceptance bar (max|err| <= 1e-2 max|ref|, relative
Frobenius <= 5e-3)."""
import numpy as np
import pytest

from paper_2405_03594_gb300 import synth
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


class MiniStack:
    """A chained stack with its own shapes: per layer qkv [3D, D] (store), o [D, D]
    (residual on h, x = qkv[:, 2D:]), gate/up [2F, D] with interleaved rows (pair product
    into a), down [D, F] (residual on h); distinct seeded weights per layer."""

    def __init__(self, D, F, layers, pct, int8, std, seed=0, host=None):
        """host: one layer's {name: (values, mask, scale or None)} in the original row order
        (stack.host_layer); given, every layer is a device copy of it."""
        import torch

        from paper_2405_03594_gb300 import sp
        from paper_2405_03594_gb300.stack import interleave_rows

        self.D, self.F, self.layers = D, F, layers
        self.host, self.mats = [], []
        shapes = {"qkv": (3 * D, D), "o": (D, D), "gate_up": (2 * F, D), "down": (D, F)}
        for l in range(layers):
            hl, ml = {}, {}
            for p, (name, (N, K)) in enumerate(shapes.items()):
                if host is not None:
                    vals, mask, s = host[name]
                    if name == "gate_up":
                        vals, mask = interleave_rows(vals, F), interleave_rows(mask, F)
                        s = None if s is None else interleave_rows(s, F)
                    hl[name] = (vals, mask, s)
                    if l > 0:
                        ml[name] = self.mats[0][name].clone()
                        continue
                else:
                    W = synth.weight(N, K, synth.rng(seed, l, p, synth.STREAM_W), std=std)
                    mask = synth.magnitude_mask(W, pct)
                    if name == "gate_up":
                        W, mask = interleave_rows(W, F), interleave_rows(mask, F)
                    if int8:
                        q, s = synth.quantize_int8(W, mask)
                        hl[name] = (q, mask, s)
                    else:
                        hl[name] = (W, mask, None)
                vals, mask, s = hl[name]
                if s is not None:
                    ml[name] = sp.compress(gu.i8_to_dev(vals), gu.u8_to_dev(mask), gu.f32_to_dev(s))
                else:
                    ml[name] = sp.compress(gu.bf16_to_dev(vals), gu.u8_to_dev(mask))
            self.host.append(hl)
            self.mats.append(ml)
        r = synth.activations(2 * layers, D, synth.rng(seed, 0, 9, synth.STREAM_RESID))
        self.r = [gu.bf16_to_dev(r[i]) for i in range(2 * layers)]
        self.r_host = r
        bf = dict(dtype=torch.bfloat16, device="cuda")
        self.h = torch.zeros((4, D), **bf)
        self.qkv = torch.zeros((4, 3 * D), **bf)
        self.a = torch.zeros((4, F), **bf)

    def ops(self, M):
        h, qkv, a = self.h[:M], self.qkv[:M], self.a[:M]
        out = []
        for l in range(self.layers):
            m = self.mats[l]
            out.append(("qkv", l, (m["qkv"], h, qkv, "store", None)))
            out.append(("o", l, (m["o"], qkv[:, 2 * self.D:], h, "residual", self.r[2 * l])))
            out.append(("gate_up", l, (m["gate_up"], h, a, "pair_product", None)))
            out.append(("down", l, (m["down"], a, h, "residual", self.r[2 * l + 1])))
        return out

    def reset(self, x0):
        import torch

        M = x0.shape[0]
        self.h[:M].copy_(gu.bf16_to_dev(x0))
        self.qkv.fill_(float("nan"))
        self.a.fill_(float("nan"))
        torch.cuda.synchronize()

    def state(self, M):
        return {"h": gu.bf16_bits_from_dev(self.h[:M]).copy(), "qkv": gu.bf16_bits_from_dev(self.qkv[:M]).copy(),
                "a": gu.bf16_bits_from_dev(self.a[:M]).copy()}


def _lin(oracle, host, x_bits, rows=None):
    vals, mask, s = host
    if rows is not None:
        vals, mask = vals[rows], mask[rows]
        s = None if s is None else s[rows]
    if s is not None:
        return oracle.linear_int8(x_bits, vals, mask, s)
    return oracle.linear_bf16(x_bits, vals, mask)


def _f(bits):
    return synth.bf16_to_f32(bits).astype(np.float64)


def check_chain_prefixes(st, oracle, M, x0, sample=None, seed=0):
    """Run the chain cut to k = 1 .. n linears from the same start; check linear k-1 from
    the state the cut-to-(k-1) chain left.  sample: output rows (per linear) to check."""
    from paper_2405_03594_gb300 import sp

    ops = st.ops(M)
    st.reset(x0)
    prev = st.state(M)
    g = np.random.default_rng(seed)
    for k in range(1, len(ops) + 1):
        st.reset(x0)
        sp.Chain([o for _, _, o in ops[:k]], M).run()
        sp.check()
        cur = st.state(M)
        name, l, _ = ops[k - 1]
        host = st.host[l][name]
        N = host[0].shape[0]
        what = f"linear {k - 1} ({name}, layer {l}) M={M}"
        if name == "qkv":
            rows = np.arange(N) if sample is None else np.sort(g.choice(N, sample, replace=False))
            gu.assert_close(_f(cur["qkv"])[:, rows], _lin(oracle, host, prev["h"], rows), what)
        elif name in ("o", "down"):
            xin = prev["qkv"][:, 2 * st.D:] if name == "o" else prev["a"]
            rows = np.arange(N) if sample is None else np.sort(g.choice(N, sample, replace=False))
            r = _f(st.r_host[2 * l + (0 if name == "o" else 1)])
            ref = _f(prev["h"])[:, rows] + _lin(oracle, host, np.ascontiguousarray(xin), rows) + r[rows]
            gu.assert_close(_f(cur["h"])[:, rows], ref, what)
        else:  # gate_up, pair product
            F = N // 2
            j = np.arange(F) if sample is None else np.sort(g.choice(F, sample, replace=False))
            rows = np.stack([2 * j, 2 * j + 1], axis=1).reshape(-1)
            y = _lin(oracle, host, prev["h"], rows)
            ref = y[:, 0::2] * y[:, 1::2]
            gu.assert_close(_f(cur["a"])[:, j], ref, what)
        prev = cur
    return prev


@pytest.mark.parametrize("int8", [False, True])
@pytest.mark.parametrize("M", [1, 2, 3, 4])
def test_chain_each_linear_small_ragged(oracle, M, int8):
    """D = 264, F = 200: ragged row blocks and K-tiles in every linear, 3 layers."""
    st = MiniStack(D=264, F=200, layers=3, pct=70, int8=int8, std=0.05, seed=M)
    x0 = synth.activations(M, 264, synth.rng(1, 0, 0, synth.STREAM_X))
    check_chain_prefixes(st, oracle, M, x0, seed=M)


@pytest.fixture(scope="module")
def llama_host():
    """One seeded Llama-2-7B layer at 70% (stack weight scale), bf16 and INT8 (q, s) from
    the same weights, in the original row order."""
    from paper_2405_03594_gb300.stack import host_layer

    bf = host_layer(70, False)
    i8 = {}
    for name, (W, mask, _) in bf.items():
        q, s = synth.quantize_int8(W, mask)
        i8[name] = (q, mask, s)
    return {"bf16": bf, "int8": i8}


@pytest.mark.parametrize("dt,M,layers", [("bf16", 1, 2), ("bf16", 4, 1), ("int8", 3, 1)])
def test_chain_each_linear_llama_shapes(oracle, llama_host, dt, M, layers):
    """Llama-2-7B layers (qkv 4096->12288, o, gate/up 4096->22016, down 11008->4096) at 70%:
    every CTA takes several chunks of every linear and split-K fix-ups run; the second
    layer reads what the first wrote.  384 sampled output rows (pairs for gate/up) per
    linear."""
    st = MiniStack(D=4096, F=11008, layers=layers, pct=70, int8=dt == "int8", std=None, seed=7,
                   host=llama_host[dt])
    x0 = synth.activations(M, 4096, synth.rng(2, 0, 0, synth.STREAM_X))
    check_chain_prefixes(st, oracle, M, x0, sample=384, seed=M)


def test_chain_complete_row_blocks_and_long_k(oracle):
    """Shapes that reach the other work splits: a K = 64 linear (one K-tile, so every chunk
    is a whole row block; 700 row blocks over the CTAs), then a K = 89600 linear (1400
    K-tiles, each row block summed from hundreds of CTAs' partials), then a pair product."""
    import torch

    from paper_2405_03594_gb300 import sp

    M = 3
    g = np.random.default_rng(11)
    specs = [(89600, 64, "store"), (512, 89600, "pair_product"), (640, 256, "store")]
    mats, host, ys = [], [], []
    x0 = synth.activations(M, 64, g)
    xin = gu.bf16_to_dev(x0)
    x = xin
    ops = []
    for N, K, epi in specs:
        W = synth.weight(N, K, g, std=0.1 if K < 1000 else 0.01)
        mask = synth.magnitude_mask(W, 70)
        h = sp.compress(gu.bf16_to_dev(W), gu.u8_to_dev(mask))
        ny = N // 2 if epi == "pair_product" else N
        y = torch.full((M, ny), float("nan"), dtype=torch.bfloat16, device="cuda")
        ops.append((h, x, y, epi, None))
        mats.append(h)
        host.append((W, mask))
        ys.append(y)
        x = y
    sp.Chain(ops, M).run()
    sp.check()
    xb = x0
    for (W, mask), y, (N, K, epi) in zip(host, ys, specs):
        ref = oracle.linear_bf16(xb, W, mask)
        if epi == "pair_product":
            ref = ref[:, 0::2] * ref[:, 1::2]
        got_bits = gu.bf16_bits_from_dev(y)
        gu.assert_close(_f(got_bits), ref, f"{N}x{K} {epi}")
        xb = got_bits


def test_chain_repeatable_and_leaves_workspace_clear():
    import torch

    from paper_2405_03594_gb300 import sp

    st = MiniStack(D=1024, F=2752, layers=2, pct=70, int8=False, std=0.01, seed=3)
    M = 2
    x0 = synth.activations(M, 1024, synth.rng(3, 0, 0, synth.STREAM_X))
    c = sp.Chain([o for _, _, o in st.ops(M)], M)
    outs = []
    for _ in range(3):
        st.reset(x0)
        c.run()
        sp.check()
        outs.append(st.state(M))
        assert int(torch.count_nonzero(c.workspace[:4096]).item()) == 0  # counters back at zero
    for o in outs[1:]:
        for key in o:
            assert np.array_equal(o[key], outs[0][key]), key


def test_chain_matches_per_linear_graph_path(llama_host):
    """The chained step against the same step from separate sp_linear launches and glue
    kernels (LinearStack; its gate/up weight is not interleaved): equal within tolerance."""
    import torch

    from paper_2405_03594_gb300 import sp
    from paper_2405_03594_gb300.stack import ChainStack, LinearStack

    M = 4
    ls = LinearStack(layers=2, pct=70, int8=True, max_m=4, host=llama_host["int8"])
    cs = ChainStack(layers=2, pct=70, int8=True, max_m=4, host=llama_host["int8"])
    x = gu.bf16_to_dev(synth.activations(M, 4096, synth.rng(0, 8, 0, synth.STREAM_X)))
    ls.set_input(x)
    cs.set_input(x)
    ls.step(M, reset=True)
    cs.step(M, reset=True)
    sp.check()
    a, b = gu.bf16_from_dev(cs.h[:M]), gu.bf16_from_dev(ls.h[:M])
    assert np.isfinite(a).all()
    gu.assert_close(a, b, "chain vs per-linear step")
    torch.cuda.synchronize()


def test_chain_argument_errors():
    import torch

    from paper_2405_03594_gb300 import sp

    st = MiniStack(D=264, F=200, layers=1, pct=70, int8=False, std=0.05)
    ops = [o for _, _, o in st.ops(4)]
    # more than four batch rows
    c = sp.Chain(ops, 4)
    c.m = 5
    with pytest.raises(sp.SpError) as e:
        c.run()
    assert e.value.code == 2  # SP_ERR_UNSUPPORTED
    # a workspace that is too small
    c = sp.Chain(ops, 4)
    c.workspace = torch.zeros(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(sp.SpError) as e:
        c.run()
    assert e.value.code == 8  # SP_ERR_WORKSPACE
    # an unknown epilogue
    c = sp.Chain(ops, 4)
    c._ops[1].epilogue = 7
    with pytest.raises(sp.SpError) as e:
        c.run()
    assert e.value.code == 1  # SP_ERR_INVALID_ARG
    # m == 0: nothing to do
    c = sp.Chain(ops, 4)
    c.m = 0
    c.run()
    sp.check()


def test_chain_longer_than_one_launch(oracle):
    """164 linears (41 small layers): sp_chain_run splits them into launches of at most 160;
    the linears on both sides of the split are checked from the GPU's own state, so the
    second launch must see everything the first one wrote."""
    from paper_2405_03594_gb300 import sp

    M = 2
    st = MiniStack(D=64, F=96, layers=41, pct=70, int8=False, std=0.02, seed=5)
    ops = st.ops(M)
    assert len(ops) == 164
    x0 = synth.activations(M, 64, synth.rng(4, 0, 0, synth.STREAM_X))

    def state_after(k):
        st.reset(x0)
        if k:
            sp.Chain([o for _, _, o in ops[:k]], M).run()
            sp.check()
        return st.state(M)

    prev = state_after(158)
    for k in (159, 160, 161, 162):
        cur = state_after(k)
        name, l, _ = ops[k - 1]
        host = st.host[l][name]
        what = f"linear {k - 1} ({name}, layer {l})"
        if name == "qkv":
            gu.assert_close(_f(cur["qkv"]), _lin(oracle, host, prev["h"]), what)
        elif name in ("o", "down"):
            xin = prev["qkv"][:, 2 * st.D:] if name == "o" else prev["a"]
            r = _f(st.r_host[2 * l + (0 if name == "o" else 1)])
            ref = _f(prev["h"]) + _lin(oracle, host, np.ascontiguousarray(xin)) + r
            gu.assert_close(_f(cur["h"]), ref, what)
        else:
            y = _lin(oracle, host, prev["h"])
            gu.assert_close(_f(cur["a"]), y[:, 0::2] * y[:, 1::2], what)
        prev = cur
