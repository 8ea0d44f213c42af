"""af1_step_*: a decode step of many linears in dependent levels as one
persistent launch, against the FP64 oracle through the C ABI.

Each linear's output is compared with the oracle evaluated on exactly the
FP16 input that linear read (for chained linears: the FP16 output of its
producer, as stored by the step), within the row-wise relative error bar;
integer-exact steps must match bit for bit."""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, f16, oracle_from_signs, signs_layer, words_layer

pytestmark = pytest.mark.gpu

# A LLaMA-3-8B decoder layer: (name, d_out, d_in) and its level in the
# decoder's dependency order (q | k | v, o, gate | up, down).
LAYER = [("q", 4096, 4096, 0), ("k", 1024, 4096, 0), ("v", 1024, 4096, 0), ("o", 4096, 4096, 1),
         ("gate", 14336, 4096, 2), ("up", 14336, 4096, 2), ("down", 4096, 14336, 3)]


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


def _pad(n, align=8):
    return n + (-n) % align


def _ybuf(tokens, m, dtype):
    return torch.zeros((tokens, _pad(m, 8 if dtype == torch.float16 else 4)), dtype=dtype, device="cuda")


def _xbuf(bits, tokens, n):
    x = torch.zeros((tokens, _pad(n)), dtype=torch.float16, device="cuda")
    x[:, :n] = f16(bits).reshape(tokens, n)
    return x


def _run(P, step, ws=None, times=1):
    ws = step.make_workspace() if ws is None else ws
    for _ in range(times):
        step.run(ws)
    torch.cuda.synchronize()
    P.workspace_status(ws)
    return ws


@pytest.mark.parametrize("tokens", [1, 2, 3, 4])
def test_decoder_layer_independent_inputs(P, tokens):
    layers, items, refs = [], [], []
    for i, (name, m, n, level) in enumerate(LAYER):
        r = O.rank_for_budget(m, n, 1)
        d = synth.layer_words(500 + 10 * i + tokens, m, n, r, tokens)
        L = words_layer(P, d, m, n, r)
        x = _xbuf(d["x"], tokens, n)
        y = _ybuf(tokens, m, torch.float32)
        layers.append(L)
        items.append((L, x, y, level))
        rows = np.sort(synth.rng(i).choice(m, size=min(m, 384), replace=False))
        refs.append((y, rows, O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r,
                                                    rows=rows), m))
    step = P.Step(items)
    info = step.info()
    assert info["levels"] == 4 and info["ctas"] >= 152
    _run(P, step)
    for (y, rows, ref, m) in refs:
        got = y[:tokens, :m].double().cpu().numpy()[:, rows]
        assert O.rowwise_rel_err(got, ref) <= TOL
    step.destroy()
    for L in layers:
        L.free()


def _chain_layer(P, seed, m, n, r):
    """A layer whose gain keeps activations of order one: a, b ~ U(0.5, 1.5),
    s ~ U(0.5, 1.5) / sqrt(n r)."""
    g = synth.rng(seed)
    U = synth.signs(g, m, r)
    V = synth.signs(g, n, r)
    a = synth.unit_gain_scales_f16(g, m, 1.0)
    s = synth.unit_gain_scales_f16(g, r, 1.0 / np.sqrt(n * r))
    b = synth.unit_gain_scales_f16(g, n, 1.0)
    d = dict(U=U, V=V, a=a, s=s, b=b)
    return d, signs_layer(P, d)


@pytest.mark.parametrize("tokens", [1, 2])
def test_chained_decoder_layers_with_swiglu(P, tokens):
    """Two decoder layers whose linears read each other's outputs: q, k, v
    read the layer input, o reads q, gate and up read o, down reads
    h = FP16(SiLU(gate) up), and the next layer's q, k, v read down's output.
    Smaller LLaMA-like widths (d = 1024, d_ff = 2816) keep the oracle quick."""
    d_model, d_ff = 1024, 2816
    shapes = {"q": (d_model, d_model), "k": (256, d_model), "v": (256, d_model), "o": (d_model, d_model),
              "gate": (d_ff, d_model), "up": (d_ff, d_model), "down": (d_model, d_ff)}
    g = synth.rng(77 + tokens)
    x0_bits = synth.activations_f16(g, tokens, d_model)
    x0 = _xbuf(x0_bits, tokens, d_model)
    items, recs, layers = [], [], []
    cur = x0
    for layer_i in range(2):
        outs = {}
        for j, name in enumerate(["q", "k", "v", "o", "gate", "up", "down"]):
            m, n = shapes[name]
            r = O.rank_for_budget(m, n, 1)
            d, L = _chain_layer(P, 1000 * layer_i + j, m, n, r)
            layers.append(L)
            y = _ybuf(tokens, m, torch.float16)
            level = 4 * layer_i + {"q": 0, "k": 0, "v": 0, "o": 1, "gate": 2, "up": 2, "down": 3}[name]
            if name in ("q", "k", "v"):
                x, x2 = cur, None
            elif name == "o":
                x, x2 = outs["q"], None
            elif name in ("gate", "up"):
                x, x2 = outs["o"], None
            else:
                x, x2 = outs["gate"], outs["up"]
            items.append((L, x, y, level) if x2 is None else (L, x, y, level, x2))
            recs.append((name, d, m, n, r, x, x2, y))
            outs[name] = y
        cur = outs["down"]
    step = P.Step(items)
    _run(P, step)
    for (name, d, m, n, r, x, x2, y) in recs:
        xin = x[:tokens, :n].cpu().numpy().view(np.uint16)
        if x2 is not None:
            xin = O.swiglu_f16(xin, x2[:tokens, :n].cpu().numpy().view(np.uint16))
        dd = dict(d, x=xin)
        ref = oracle_from_signs(dd, n)
        got = y[:tokens, :m].double().cpu().numpy()
        assert np.abs(ref).max() > 1e-2, name  # activations stay of order one
        # FP16 output: the bar plus the output rounding (2^-11 relative)
        assert O.rowwise_rel_err(got, ref) <= TOL, name
    step.destroy()
    for L in layers:
        L.free()


def test_integer_exact_bit_for_bit(P):
    """Unit scales and integer activations: every partial sum is an exact
    integer in FP32, so the step equals the oracle bit for bit."""
    specs = [(300, 520, 200, 0), (128, 256, 129, 0), (700, 130, 77, 1), (64, 1000, 300, 2), (513, 257, 255, 2)]
    tokens = 3
    items, recs, layers = [], [], []
    for i, (m, n, r, level) in enumerate(specs):
        d = synth.integer_layer(900 + i, m, n, r, tokens)
        L = signs_layer(P, d)
        layers.append(L)
        x = _xbuf(d["x"], tokens, n)
        y = _ybuf(tokens, m, torch.float32)
        items.append((L, x, y, level))
        recs.append((d, n, m, y))
    step = P.Step(items)
    _run(P, step)
    for (d, n, m, y) in recs:
        np.testing.assert_array_equal(y[:tokens, :m].double().cpu().numpy(), oracle_from_signs(d, n))
    step.destroy()
    for L in layers:
        L.free()


def test_ragged_shapes_many_levels_and_reuse(P):
    """Shapes that are not multiples of 128, five levels, FP16 outputs; three
    runs on one workspace give identical bits (counters reset, fixed
    summation order)."""
    specs = [(100, 130, 77), (1000, 700, 321), (520, 2000, 600), (33, 70, 31), (257, 129, 200)]
    tokens = 2
    items, recs, layers = [], [], []
    for i, (m, n, r) in enumerate(specs):
        d = synth.layer_signs(300 + i, m, n, r, tokens)
        L = signs_layer(P, d)
        layers.append(L)
        x = _xbuf(d["x"], tokens, n)
        y = _ybuf(tokens, m, torch.float16)
        items.append((L, x, y, i))
        recs.append((d, n, m, y))
    step = P.Step(items)
    ws = step.make_workspace()
    outs = []
    for _ in range(3):
        _run(P, step, ws)
        outs.append([y[:tokens, :m].clone() for (_d, _n, m, y) in recs])
    for (d, n, m, y) in recs:
        assert O.rowwise_rel_err(y[:tokens, :m].double().cpu().numpy(), oracle_from_signs(d, n)) <= TOL
    for a, b in zip(outs[0], outs[2]):
        assert torch.equal(a, b)
    step.destroy()
    for L in layers:
        L.free()


def test_step_matches_per_call_path(P):
    """The step and af1_linear_forward agree per linear (both within the bar
    of the oracle; here directly against each other)."""
    tokens = 1
    items, recs, layers = [], [], []
    for i, (name, m, n, level) in enumerate(LAYER[:4]):
        r = O.rank_for_budget(m, n, 1)
        d = synth.layer_words(700 + i, m, n, r, tokens)
        L = words_layer(P, d, m, n, r)
        layers.append(L)
        x = _xbuf(d["x"], tokens, n)
        y = _ybuf(tokens, m, torch.float32)
        items.append((L, x, y, level))
        recs.append((L, x, y, m))
    step = P.Step(items)
    _run(P, step)
    for (L, x, y, m) in recs:
        ref = L.forward(x, out_dtype=torch.float32)
        torch.cuda.synchronize()
        assert O.rowwise_rel_err(y[:, :m].double().cpu().numpy(), ref.double().cpu().numpy()) <= 1e-5
    step.destroy()
    for L in layers:
        L.free()


def test_gate_wait_times_out_then_recovers(P):
    """A step whose level 0 waits for a gate word that nobody opens: with a
    short wait budget every wait gives up, the status reports
    AF1_ERR_TIMEOUT and the counters are reset, so the next run with the gate
    opened matches the oracle on the same workspace."""
    specs = [(256, 512, 200, 0), (300, 256, 100, 1)]
    tokens = 1
    items, recs, layers = [], [], []
    for i, (m, n, r, level) in enumerate(specs):
        d = synth.layer_signs(50 + i, m, n, r, tokens)
        L = signs_layer(P, d)
        layers.append(L)
        x = _xbuf(d["x"], tokens, n)
        y = _ybuf(tokens, m, torch.float32)
        items.append((L, x, y, level))
        recs.append((d, n, m, y))
    step = P.Step(items, gate=True)
    ws = step.make_workspace()
    old = P.get_wait_cycles()
    try:
        P.set_wait_cycles(100000)  # about 50 us
        step.run(ws)
        torch.cuda.synchronize()
        with pytest.raises(P.AF1Error) as ei:
            P.workspace_status(ws)
        assert ei.value.code == -7
        P.workspace_status(ws)  # the report cleared the status word
    finally:
        P.set_wait_cycles(old)
    P.Step.open_gate(ws)
    _run(P, step, ws)
    for (d, n, m, y) in recs:
        assert O.rowwise_rel_err(y[:tokens, :m].double().cpu().numpy(), oracle_from_signs(d, n)) <= TOL
    step.destroy()
    for L in layers:
        L.free()


def test_full_hisa_stack_sampled_rows(P):
    """The 32-layer LLaMA-3-8B-shaped stack with HiSA-like ranks (+-30 %
    around each matrix's 1.0-BPW rank, renormalised to 1.0 BPW), one token,
    each linear's output checked on sampled rows against the oracle."""
    import bench
    names = [(m, n) for _ in range(32) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    ranks = bench.hisa_ranks(names)
    levels = [0, 0, 0, 1, 2, 2, 3]
    items, recs, layers = [], [], []
    for i, ((m, n), r) in enumerate(zip(names, ranks)):
        d = synth.layer_words(20000 + i, m, n, r, 1)
        L = words_layer(P, d, m, n, r)
        layers.append(L)
        x = _xbuf(d["x"], 1, n)
        y = _ybuf(1, m, torch.float16)
        items.append((L, x, y, 4 * (i // 7) + levels[i % 7]))
        recs.append((d, m, n, r, y))
    step = P.Step(items)
    assert step.info()["levels"] == 128
    _run(P, step, times=2)
    for i, (d, m, n, r, y) in enumerate(recs):
        if i % 5 != 0 and i % 7 != 6:
            continue  # a sample of the linears, every down projection among them
        rows = np.sort(synth.rng(i).choice(m, size=64, replace=False))
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
        assert O.rowwise_rel_err(y[:1, :m].double().cpu().numpy()[:, rows], ref) <= TOL, i
    step.destroy()
    for L in layers:
        L.free()
