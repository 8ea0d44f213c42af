"""af1_linear_forward_swiglu against the FP64 oracle, through the C ABI: the
down projection of a LLaMA MLP fed h = FP16(SiLU(g) * u) from the gate and
up outputs. Decode passes on the CUDA-core kernels (clustered and streaming)
form h while staging; the tensor-core decode and the prefill path form it in
the workspace first."""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, f16, oracle_from_signs, signs_layer, words_layer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


def _gu(seed, tokens, n):
    g = synth.rng(seed)
    return synth.activations_f16(g, tokens, n), synth.activations_f16(g, tokens, n)


def _run(layer, gb, ub, n, out_dtype=torch.float32):
    gt = f16(gb).reshape(-1, n)
    ut = f16(ub).reshape(-1, n)
    y = layer.forward_swiglu(gt, ut, out_dtype=out_dtype)
    torch.cuda.synchronize()
    return y.double().cpu().numpy()


@pytest.mark.parametrize("m,n,r", [(100, 130, 77), (1000, 700, 321), (300, 1920, 100)])
@pytest.mark.parametrize("tokens", [1, 2, 5, 16, 40])
@pytest.mark.parametrize("path", ["default", "stream", "tc"])
def test_swiglu_matches_oracle(P, m, n, r, tokens, path):
    if path == "stream" and tokens > 2:
        pytest.skip("the streaming kernel takes passes of 1-2 tokens")
    d = synth.layer_signs(5 * m + n + tokens, m, n, r, 1)
    layer = signs_layer(P, d, stream_decode=path == "stream", tc_decode=path == "tc")
    gb, ub = _gu(m + tokens, tokens, n)
    y = _run(layer, gb, ub, n)
    d["x"] = O.swiglu_f16(gb, ub)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("tokens", [1, 3, 16])
@pytest.mark.parametrize("path", ["default", "stream", "tc"])
def test_swiglu_integer_bit_exact(P, tokens, path):
    """Decode passes. g in [17, 20] (SiLU(g) = g exactly in FP32 and after
    FP16 rounding), u in {-1, 0, 1}, unit scales: h and y are integers the
    kernels must hit bit for bit (any mix-up of g and u columns or rows
    shows)."""
    if path == "stream" and tokens > 2:
        pytest.skip("the streaming kernel takes passes of 1-2 tokens")
    m, n, r = 256, 96, 40
    d = synth.integer_layer(41 + tokens, m, n, r, 1)
    rg = synth.rng(tokens)
    gb = rg.integers(17, 21, size=(tokens, n)).astype(np.float16).view(np.uint16)
    ub = rg.integers(-1, 2, size=(tokens, n)).astype(np.float16).view(np.uint16)
    layer = signs_layer(P, d, stream_decode=path == "stream", tc_decode=path == "tc")
    y = _run(layer, gb, ub, n)
    d["x"] = O.swiglu_f16(gb, ub)
    np.testing.assert_array_equal(d["x"].view(np.float16).astype(np.float64),
                                  (gb.view(np.float16).astype(np.float64) * ub.view(np.float16).astype(np.float64)))
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


def test_swiglu_prefill_two_passes(P):
    m, n, r = 200, 136, 64
    tokens = 2100  # passes of 2048 and 52 tokens
    d = synth.layer_signs(97, m, n, r, 1)
    layer = signs_layer(P, d)
    gb, ub = _gu(98, tokens, n)
    y = _run(layer, gb, ub, n, torch.float16)
    d["x"] = O.swiglu_f16(gb, ub)
    assert O.rowwise_rel_err(y, oracle_from_signs(d, n)) <= TOL
    layer.free()


@pytest.mark.parametrize("m,n", [(4096, 14336), (8192, 28672)])
@pytest.mark.parametrize("tokens", [1, 16])
def test_swiglu_full_size_down_projection(P, m, n, tokens):
    """Down projections of LLaMA-3-8B and LLaMA-70B at the 1.0-BPW rank."""
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(31 + m // 1024 + tokens, m, n, r, 1)
    layer = words_layer(P, d, m, n, r)
    gb, ub = _gu(7 + tokens, tokens, n)
    y = _run(layer, gb, ub, n)
    rows = np.sort(synth.rng(tokens).choice(m, size=256, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], O.swiglu_f16(gb, ub), m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


def test_swiglu_errors(P):
    m, n, r = 64, 96, 40
    d = synth.layer_signs(3, m, n, r, 1)
    layer = signs_layer(P, d)
    g = torch.zeros((2, n), dtype=torch.float16, device="cuda")
    u = torch.zeros((2, n + 8), dtype=torch.float16, device="cuda")
    y = torch.empty((2, m), dtype=torch.float32, device="cuda")
    ws = torch.zeros(layer.workspace_bytes_swiglu(2), dtype=torch.uint8, device="cuda")
    assert layer.workspace_bytes_swiglu(2) > layer.workspace_bytes(2)
    with pytest.raises(P.AF1Error) as e:  # u 2 bytes past a 16-byte boundary
        P._check(P._lib.af1_linear_forward_swiglu(layer._h, g.data_ptr(), u.data_ptr() + 2, n, 2, y.data_ptr(), m,
                                                  P.AF1_F32, ws.data_ptr(), ws.numel(), None))
    assert e.value.code == -3
    small = torch.zeros(layer.workspace_bytes(2), dtype=torch.uint8, device="cuda")
    with pytest.raises(P.AF1Error) as e:
        layer.forward_swiglu_into(g, torch.zeros_like(g), y, small)
    assert e.value.code == -8
    layer.free()
