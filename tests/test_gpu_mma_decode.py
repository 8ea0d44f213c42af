"""The 16-bit-operand tensor-core decode kernel (AF1_FLAG_MMA_DECODE; by
default the kernel of passes of 5..16 tokens, and of calls of 17..64 tokens
as one pass) against the FP64 oracle, through the C ABI.

Phase 1 multiplies exact +-b_j FP16 sign values with the FP16 activations,
phase 2 exact +-1 BF16 values with s' split into two BF16 terms (N = 16 or
32 rows of B for up to 8 and 16 tokens). The cases cover every B
width, ragged shapes (rows and columns that end inside a chunk, ranks that
are not multiples of 128), clusters of 1..16 CTAs, K slices longer than the
tensor-memory ring, integer inputs bit for bit, the LLaMA-3-8B and 70B-class
shapes at full size on sampled rows, and the dispatch between this kernel
and the lookup tables.
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


@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (100, 130, 77), (256, 384, 200), (1000, 700, 321),
                                   (1024, 4096, 800), (300, 1920, 100)])
@pytest.mark.parametrize("tokens", [1, 2, 3, 4, 5, 6, 10, 11, 16])
def test_mma_decode_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(13 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, mma_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("m,n,r", [(64, 96, 40), (256, 256, 120), (700, 900, 333)])
@pytest.mark.parametrize("tokens", [1, 7, 12, 16])
def test_mma_decode_integer_bit_exact(P, m, n, r, tokens):
    """Unit scales and integer activations: every product and partial sum is
    an integer below 2^24, and s' (an integer below 2^16 here) is held
    exactly by its two BF16 terms, so the result is the oracle's bit for bit."""
    d = synth.integer_layer(17 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, mma_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


def test_mma_decode_fp16_output_and_outliers(P):
    """FP16 outputs, and activations with 1 % of the channels x20."""
    m, n, r, tokens = 1024, 4096, 800, 9
    d = synth.layer_signs(606, m, n, r, tokens, outlier_frac=0.01)
    layer = signs_layer(P, d, mma_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float16)
    assert O.rowwise_rel_err(y, oracle_from_signs(d, n)) <= TOL
    layer.free()


@pytest.mark.parametrize("m,n", [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336)])
@pytest.mark.parametrize("tokens", [5, 8, 16])
def test_mma_decode_llama_shapes_sampled_rows(P, m, n, tokens):
    """Default dispatch at 5..16 tokens on the LLaMA-3-8B shapes (exact
    1.0-BPW ranks), sampled rows against the oracle."""
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(31 + m // 1024 + n // 1024 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(tokens + 5).choice(m, size=256, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


@pytest.mark.parametrize("m,n", [(8192, 8192), (1024, 8192), (28672, 8192), (8192, 28672)])
def test_mma_decode_70b_shapes_8_tokens(P, m, n):
    """The 70B-class shapes at 8 tokens (the decode side of the
    decode/prefill crossover), sampled rows against the oracle."""
    tokens = 8
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(57 + m // 1024 + n // 1024, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(m + n).choice(m, size=192, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


@pytest.mark.parametrize("m,n,r,tokens,kernel", [(1000, 700, 321, 4, "lut"), (4096, 4096, 1024, 4, "lut"),
                                                  (1000, 700, 321, 5, "mma"), (1000, 700, 321, 16, "mma")])
def test_default_dispatch_matches_forced_kernels(P, m, n, r, tokens, kernel):
    """The default dispatch: passes of more than 4 tokens take the
    16-bit-operand kernel, passes of 1-4 tokens the lookup tables. The
    default result is bit-identical to the expected kernel's (forced by its
    flag), and both kernels are within the bar of the oracle."""
    d = synth.layer_signs(808 + tokens + m, m, n, r, tokens)
    ys = {}
    for kind, kw in (("default", {}), ("mma", {"mma_decode": True}), ("lut", {"lut_decode": True})):
        layer = signs_layer(P, d, **kw)
        ys[kind] = run_gpu(layer, d["x"], n)
        layer.free()
    np.testing.assert_array_equal(ys["default"], ys[kernel])
    ref = oracle_from_signs(d, n)
    assert O.rowwise_rel_err(ys["lut"], ref) <= TOL
    assert O.rowwise_rel_err(ys["mma"], ref) <= TOL


def test_mma_decode_repeatable_and_workspace_reuse(P):
    """Two layers sharing one workspace, called alternately: every call gives
    the same bits (no state is carried between calls)."""
    tokens = 11
    ds = [synth.layer_signs(900 + i, 700, 896, 333, tokens) for i in range(2)]
    layers = [signs_layer(P, d, mma_decode=True) for d in ds]
    ws = layers[0].make_workspace(tokens)
    assert ws.numel() >= layers[1].make_workspace(tokens).numel()
    xs = [f16(d["x"]).reshape(tokens, 896) for d in ds]
    outs = []
    for rep in range(2):
        for L, x in zip(layers, xs):
            y = torch.empty((tokens, 700), dtype=torch.float32, device="cuda")
            L.forward_into(x, y, ws)
            outs.append(y)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(outs[0].cpu().numpy(), outs[2].cpu().numpy())
    np.testing.assert_array_equal(outs[1].cpu().numpy(), outs[3].cpu().numpy())
    for d, y in zip(ds, outs[:2]):
        assert O.rowwise_rel_err(y.double().cpu().numpy(), oracle_from_signs(d, 896)) <= TOL
    for L in layers:
        L.free()


def test_decode_kernel_flags_exclusive(P):
    d = synth.layer_signs(54, 64, 96, 20, 1)
    for kw in ({"tc_decode": True, "mma_decode": True}, {"mma_decode": True, "lut_decode": True},
               {"tc_decode": True, "lut_decode": True}):
        with pytest.raises(P.AF1Error):
            signs_layer(P, d, **kw)


# ---------------------------------------------------------------------------
# Passes of 17..64 tokens on the same kernel (one pass instead of the prefill
# kernel): B of up to 64 rows in phase 1 and 128 in phase 2.
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("m,n,r", [(100, 130, 77), (1000, 700, 321), (1024, 4096, 800), (300, 1920, 100)])
@pytest.mark.parametrize("tokens", [17, 24, 32, 33, 48, 64])
def test_mid_pass_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(23 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n, torch.float32)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("m,n,r", [(256, 256, 120), (700, 896, 333)])
@pytest.mark.parametrize("tokens", [20, 64])
def test_mid_pass_integer_bit_exact(P, m, n, r, tokens):
    d = synth.integer_layer(29 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


@pytest.mark.parametrize("tokens", [17, 64])
def test_mid_pass_against_prefill_path(P, tokens):
    """The same layer with AF1_FLAG_TC_DECODE runs calls of more than 16
    tokens on the prefill kernel instead: both within the bar of the oracle,
    FP16 outputs with x20 outlier channels."""
    m, n, r = 1024, 4096, 800
    d = synth.layer_signs(4040 + tokens, m, n, r, tokens, outlier_frac=0.01)
    ref = oracle_from_signs(d, n)
    for kw in ({}, {"tc_decode": True}):
        layer = signs_layer(P, d, **kw)
        y = run_gpu(layer, d["x"], n, torch.float16)
        assert O.rowwise_rel_err(y, ref) <= TOL, kw
        layer.free()


@pytest.mark.parametrize("m,n,tokens", [(4096, 14336, 20), (8192, 8192, 32), (4096, 4096, 64), (1024, 8192, 48)])
def test_mid_pass_full_size_sampled_rows(P, m, n, tokens):
    """Full-size matrices that take one pass at these widths (up to 32
    tokens below 70 M signs, up to 64 below 20 M)."""
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(61 + m // 1024 + n // 1024, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(m + n + tokens).choice(m, size=128, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()
