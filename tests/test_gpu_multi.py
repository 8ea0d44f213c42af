"""Several layers sharing one input (af1_linear_forward_multi) against the
FP64 oracle per layer, through the C ABI."""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, f16, oracle_from_signs, signs_layer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


def _group(P, seed, n, specs, tokens, integer=False):
    """Layers (m_i, r_i) with input width n and one shared x."""
    ds, layers = [], []
    for i, (m, r) in enumerate(specs):
        if integer:
            d = synth.integer_layer(seed + i, m, n, r, tokens)
        else:
            d = synth.layer_signs(seed + i, m, n, r, tokens)
        ds.append(d)
        layers.append(signs_layer(P, d))
    x = ds[0]["x"]  # every layer gets the first layer's activations
    for d in ds:
        d["x"] = x
    return ds, layers, x


def _run(P, layers, x_bits, n, tokens, out_dtype=torch.float32):
    x = f16(x_bits).reshape(tokens, n)
    pad = (-n) % 8
    xp = torch.zeros((tokens, n + pad), dtype=torch.float16, device="cuda")
    xp[:, :n] = x
    ys = []
    for L in layers:
        align = 8 if out_dtype == torch.float16 else 4
        ys.append(torch.full((tokens, L.m + (-L.m) % align), float("nan"), dtype=out_dtype, device="cuda"))
    ws = torch.zeros(P.workspace_bytes_multi(layers, tokens), dtype=torch.uint8, device="cuda")
    P.forward_multi(layers, xp, ys, ws)
    P.workspace_status(ws)
    torch.cuda.synchronize()
    return [y[:, :L.m].double().cpu().numpy() for L, y in zip(layers, ys)]


@pytest.mark.parametrize("specs", [[(200, 77), (100, 40), (100, 40)], [(300, 120), (64, 30)],
                                   [(256, 200), (129, 60), (64, 33), (1000, 321)], [(520, 600)]])
@pytest.mark.parametrize("tokens", [1, 3, 5, 8, 16, 17])
def test_multi_matches_oracle(P, specs, tokens):
    n = 700
    ds, layers, x = _group(P, 40 + tokens + len(specs), n, specs, tokens)
    ys = _run(P, layers, x, n, tokens)
    for d, y in zip(ds, ys):
        err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
        assert err <= TOL, err
    for L in layers:
        L.free()


@pytest.mark.parametrize("tokens", [1, 4, 7, 16])
def test_multi_integer_bit_exact(P, tokens):
    n = 256
    ds, layers, x = _group(P, 70 + tokens, n, [(130, 100), (64, 40), (200, 120)], tokens, integer=True)
    ys = _run(P, layers, x, n, tokens)
    for d, y in zip(ds, ys):
        np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    for L in layers:
        L.free()


@pytest.mark.parametrize("tokens", [1, 4, 16])
def test_multi_single_layer_identical(P, tokens):
    """count == 1 runs exactly the kernels of af1_linear_forward."""
    n = 4096
    d = synth.layer_signs(90 + tokens, 1024, n, 800, tokens)
    layer = signs_layer(P, d)
    (y_multi,) = _run(P, [layer], d["x"], n, tokens)
    x = f16(d["x"]).reshape(tokens, n)
    y_one = layer.forward(x, out_dtype=torch.float32).double().cpu().numpy()
    np.testing.assert_array_equal(y_multi, y_one)
    layer.free()


def test_multi_llama_qkv_full_size(P):
    """q, k, v of a LLaMA-3-8B-shaped layer at their 1.0-BPW ranks, one token,
    sampled rows against the oracle."""
    n, tokens = 4096, 1
    specs = [(4096, O.rank_for_budget(4096, n, 1)), (1024, O.rank_for_budget(1024, n, 1)),
             (1024, O.rank_for_budget(1024, n, 1))]
    ds = [synth.layer_words(300 + i, m, n, r, tokens) for i, (m, r) in enumerate(specs)]
    from tests.af1_cases import words_layer
    layers = [words_layer(P, d, m, n, r) for d, (m, r) in zip(ds, specs)]
    ys = _run(P, layers, ds[0]["x"], n, tokens)
    for d, (m, r), y in zip(ds, specs, ys):
        rows = np.sort(synth.rng(m).choice(m, size=128, replace=False))
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], ds[0]["x"], m, n, r, rows=rows)
        assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    for L in layers:
        L.free()


@pytest.mark.parametrize("specs", [[(200, 77), (100, 40), (100, 40)], [(300, 120), (64, 30)],
                                   [(256, 200), (129, 60), (64, 33), (1000, 321)]])
@pytest.mark.parametrize("tokens", [18, 40, 64, 129, 300])
def test_multi_prefill_matches_oracle(P, specs, tokens):
    """Passes longer than 16 tokens: each layer runs the stream-K prefill
    GEMMs from its own workspace slice, all reporting to the first slice's
    status word (ragged ranks and row counts per layer)."""
    n = 700
    ds, layers, x = _group(P, 140 + tokens + len(specs), n, specs, tokens)
    ys = _run(P, layers, x, n, tokens)
    for d, y in zip(ds, ys):
        err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
        assert err <= TOL, err
    for L in layers:
        L.free()


@pytest.mark.parametrize("tokens", [17, 100, 257])
def test_multi_prefill_integer_bit_exact_fp16_out(P, tokens):
    """Integer-valued layers through the multi-layer call at prefill sizes
    (every sum exact in FP32, H exact in FP16), FP16 outputs (the 32-token
    TMA-store chunks), twice: equal bits each time, and equal to the
    oracle's value rounded to FP16 (|y| stays far below the FP16 range)."""
    n = 512
    ds, layers, x = _group(P, 170 + tokens, n, [(300, 200), (130, 100), (64, 40)], tokens, integer=True)
    y1 = _run(P, layers, x, n, tokens, out_dtype=torch.float16)
    y2 = _run(P, layers, x, n, tokens, out_dtype=torch.float16)
    for d, a, b in zip(ds, y1, y2):
        np.testing.assert_array_equal(a, b)
        ref = oracle_from_signs(d, n)
        assert np.abs(ref).max() < 60000
        np.testing.assert_array_equal(a, ref.astype(np.float16).astype(np.float64))
    for L in layers:
        L.free()


@pytest.mark.parametrize("tokens", [64, 2048, 2100])
def test_multi_prefill_matches_single_calls(P, tokens):
    """The multi-layer call agrees with each layer's own call (up to the
    rounding of H to FP16 should the stream-K split differ), including a
    second pass of tokens, and sampled tokens match the oracle."""
    n = 1024
    specs = [(1024, 400), (256, 160), (256, 160)]
    ds, layers, x = _group(P, 190 + tokens, n, specs, tokens)
    ys = _run(P, layers, x, n, tokens)
    xt = f16(x).reshape(tokens, n)
    toks = np.sort(synth.rng(tokens).choice(tokens, size=min(tokens, 64), replace=False))
    xs = np.asarray(x).reshape(tokens, n)[toks]
    for L, y, d in zip(layers, ys, ds):
        y_one = L.forward(xt, out_dtype=torch.float32).double().cpu().numpy()
        assert O.rowwise_rel_err(y, y_one) <= 1e-3
        ref = oracle_from_signs(dict(d, x=xs), n)
        assert O.rowwise_rel_err(y[toks], ref) <= TOL
    for L in layers:
        L.free()


def test_multi_llama_qkv_prefill_full_size(P):
    """q, k, v of a LLaMA-3-8B-shaped layer at their 1.0-BPW ranks over a
    2048-token pass: sampled rows and tokens against the oracle."""
    n, tokens = 4096, 2048
    specs = [(4096, O.rank_for_budget(4096, n, 1)), (1024, O.rank_for_budget(1024, n, 1)),
             (1024, O.rank_for_budget(1024, n, 1))]
    ds = [synth.layer_words(320 + i, m, n, r, tokens) for i, (m, r) in enumerate(specs)]
    from tests.af1_cases import words_layer
    layers = [words_layer(P, d, m, n, r) for d, (m, r) in zip(ds, specs)]
    ys = _run(P, layers, ds[0]["x"], n, tokens)
    toks = np.sort(synth.rng(7).choice(tokens, size=24, replace=False))
    xs = np.asarray(ds[0]["x"]).reshape(tokens, n)[toks].reshape(-1)
    for d, (m, r), y in zip(ds, specs, ys):
        rows = np.sort(synth.rng(m).choice(m, size=96, replace=False))
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], xs, m, n, r, rows=rows)
        assert O.rowwise_rel_err(y[toks][:, rows], ref) <= TOL
    for L in layers:
        L.free()


def test_multi_errors(P):
    d1 = synth.layer_signs(95, 64, 96, 20, 1)
    d2 = synth.layer_signs(96, 64, 128, 20, 1)
    L1, L2 = signs_layer(P, d1), signs_layer(P, d2)
    x = torch.zeros((1, 96), dtype=torch.float16, device="cuda")
    y = torch.zeros((1, 64), dtype=torch.float32, device="cuda")
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    with pytest.raises(P.AF1Error) as e:
        P.forward_multi([L1, L2], x, [y, y], ws)  # different n
    assert e.value.code == -1
    with pytest.raises(P.AF1Error) as e:
        P.forward_multi([L1] * 5, x, [y] * 5, ws)  # more than 4 layers
    assert e.value.code == -1
    with pytest.raises(P.AF1Error) as e:
        P.forward_multi([L1, L1], x, [y, y], ws[:256])  # workspace too small
    assert e.value.code == -8
    L1.free()
    L2.free()


@pytest.mark.parametrize("tokens", [1, 3])
@pytest.mark.parametrize("graph", [False, True])
def test_stream_layout_keeps_results(P, tokens, graph):
    """A chain on one stream where each call reads the previous call's FP16
    output (a single layer, then another, then a multi-layer call), under
    both stream layouts. With AF1_ONE_STREAM the next kernel launches before
    its input exists and must still wait for it. Each layout repeats its own
    bits (two runs, eager and in a CUDA graph), and each link matches the
    oracle on the input it read (the layouts may split K differently, so
    they agree within the tolerance, not bit for bit)."""
    group = [(296, 400), (256, 180)]
    d0 = synth.layer_signs(1300 + tokens, 512, 1024, 300, tokens)
    d1 = synth.layer_signs(1310 + tokens, 704, 512, 250, tokens)
    l0, l1 = signs_layer(P, d0), signs_layer(P, d1)
    dg, lg, _ = _group(P, 1320 + tokens, 704, group, tokens)
    x0 = f16(d0["x"]).reshape(tokens, 1024)
    y0 = torch.empty((tokens, 512), dtype=torch.float16, device="cuda")
    y1 = torch.empty((tokens, 704), dtype=torch.float16, device="cuda")
    yg = [torch.empty((tokens, m), dtype=torch.float32, device="cuda") for (m, _r) in group]
    ws = torch.zeros(max(l0.workspace_bytes(tokens), l1.workspace_bytes(tokens),
                         P.workspace_bytes_multi(lg, tokens)), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    outs = [y0, y1] + yg

    def chain():
        l0.forward_into(x0, y0, ws, stream=s)
        l1.forward_into(y0, y1, ws, stream=s)
        P.forward_multi(lg, y1, yg, ws, stream=s)

    try:
        for layout in (P.AF1_MANY_STREAMS, P.AF1_ONE_STREAM):
            P.set_stream_layout(layout)
            g = None
            if graph:
                with torch.cuda.stream(s):
                    chain()  # warm-up outside capture
                torch.cuda.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=s):
                    chain()
            runs = []
            for _ in range(2):
                for t in outs:
                    t.fill_(float("nan"))
                if graph:
                    g.replay()
                else:
                    with torch.cuda.stream(s):
                        chain()
                torch.cuda.synchronize()
                runs.append([t.double().cpu().numpy() for t in outs])
            for a, b in zip(runs[0], runs[1]):
                np.testing.assert_array_equal(a, b)
            y0h, y1h = runs[0][0], runs[0][1]
            bits = lambda y: y.astype(np.float16).view(np.uint16)
            assert O.rowwise_rel_err(y0h, oracle_from_signs(d0, 1024)) <= TOL
            assert O.rowwise_rel_err(y1h, oracle_from_signs(dict(d1, x=bits(y0h)), 512)) <= TOL
            for d, y in zip(dg, runs[0][2:]):
                assert O.rowwise_rel_err(y, oracle_from_signs(dict(d, x=bits(y1h)), 704)) <= TOL
    finally:
        P.set_stream_layout(P.AF1_ONE_STREAM)
    P.workspace_status(ws)
    for L in [l0, l1] + lg:
        L.free()
