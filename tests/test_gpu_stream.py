"""The streaming CUDA-core decode kernel (1- and 2-token passes) against the
FP64 oracle, through the C ABI.

AF1_FLAG_STREAM_DECODE forces it wherever it has a plan, so small ragged
shapes exercise its edge cases: super rows of 1, 2 and 4 row blocks whose
last one is ragged or missing, ragged last chunks, clusters whose last CTAs
finish few or no rows, slices longer than the ring. The large
LLaMA-70B-shaped matrices take it by default.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, f16, oracle_from_signs, run_gpu, signs_layer, words_layer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


# (20000, 1000, 600) and (40000, 512, 300) plan super rows of 2 and 4 row
# blocks for the second phase (20000 and 40000 rows are not multiples of them).
@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (100, 130, 77), (300, 1920, 100), (1000, 700, 321),
                                   (1024, 4096, 800), (3000, 1000, 2500), (129, 4100, 129),
                                   (20000, 1000, 600), (40000, 512, 300)])
@pytest.mark.parametrize("tokens", [1, 2])
def test_stream_decode_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(17 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, stream_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("m,n,r", [(64, 96, 40), (256, 256, 120), (2000, 300, 256)])
@pytest.mark.parametrize("tokens", [1, 2])
def test_stream_decode_integer_bit_exact(P, m, n, r, tokens):
    d = synth.integer_layer(29 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, stream_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


def test_stream_deterministic_across_calls(P):
    """A sequence of calls on two layers and both token counts through one
    workspace: every call matches a call on a fresh workspace bit for bit."""
    ds = [synth.layer_signs(71, 3000, 1000, 700, 2), synth.layer_signs(72, 1000, 3000, 900, 2)]
    layers = [signs_layer(P, d, stream_decode=True) for d in ds]
    ws = torch.zeros(max(L.workspace_bytes(16) for L in layers), dtype=torch.uint8, device="cuda")
    for it in range(6):
        i, tokens = it % 2, 1 + (it // 2) % 2
        L, d = layers[i], ds[i]
        x = f16(d["x"]).reshape(2, -1)[:tokens].contiguous()
        y = torch.empty(tokens, L.m, dtype=torch.float32, device="cuda")
        L.forward_into(x, y, ws)
        P.workspace_status(ws)
        fresh = torch.zeros(L.workspace_bytes(tokens), dtype=torch.uint8, device="cuda")
        y2 = torch.empty_like(y)
        L.forward_into(x, y2, fresh)
        torch.cuda.synchronize()
        assert torch.equal(y, y2)
    for L in layers:
        L.free()


@pytest.mark.parametrize("m,n", [(28672, 8192), (8192, 28672)])
@pytest.mark.parametrize("tokens", [1, 2])
def test_stream_default_full_size_sampled_rows(P, m, n, tokens):
    """LLaMA-70B-shaped MLP matrices at the 1.0-BPW rank: the default plan
    streams the matrix whose clustered split needs several waves."""
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(91 + m // 1024 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(tokens + 7).choice(m, size=256, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


def test_stream_fp16_output(P):
    m, n, r = 1000, 700, 321
    d = synth.layer_signs(5, m, n, r, 2)
    layer = signs_layer(P, d, stream_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float16)
    assert O.rowwise_rel_err(y, oracle_from_signs(d, n)) <= TOL
    layer.free()


def test_stream_layers_in_multi_call(P):
    """forward_multi over layers that stream runs them one by one."""
    n, tokens = 900, 2
    specs = [(3000, 700), (1200, 500)]
    ds = [synth.layer_signs(300 + i, m, n, r, tokens) for i, (m, r) in enumerate(specs)]
    for dd in ds[1:]:
        dd["x"] = ds[0]["x"]
    layers = [signs_layer(P, dd, stream_decode=True) for dd in ds]
    x = torch.zeros((tokens, n + (-n) % 8), dtype=torch.float16, device="cuda")
    x[:, :n] = f16(ds[0]["x"]).reshape(tokens, n)
    ys = [torch.empty((tokens, L.m), dtype=torch.float32, device="cuda") for L in layers]
    ws = torch.zeros(P.workspace_bytes_multi(layers, tokens), dtype=torch.uint8, device="cuda")
    for _ in range(2):
        P.forward_multi(layers, x, ys, ws)
        P.workspace_status(ws)
        for dd, y in zip(ds, ys):
            assert O.rowwise_rel_err(y.double().cpu().numpy(), oracle_from_signs(dd, n)) <= TOL
    for L in layers:
        L.free()
