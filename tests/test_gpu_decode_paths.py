"""The decode kernels against the FP64 oracle, through the C ABI.

Decode passes (1..16 tokens) run on the CUDA-core lookup-table kernels up to
4 tokens and on the 16-bit-operand tensor-core kernel from 5 tokens on (by
default; test_gpu_mma_decode.py covers that kernel); AF1_FLAG_TC_DECODE
selects the e4m3 tensor-core kernel and AF1_FLAG_LUT_DECODE the lookup-table
kernels at every width. These cases cover the e4m3 kernel explicitly and the
lookup-table kernel at its plan's edges: clusters whose last CTA finalises a
short or empty slice of rows (14 and 15 CTAs per cluster), token groups with
a ragged last group, and the longest contraction the library accepts (32768
columns).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_oracle as O
from tests.af1_cases import TOL, oracle_from_signs, run_gpu, signs_layer, words_layer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (100, 130, 77), (256, 384, 200), (1000, 700, 321),
                                   (1024, 4096, 800)])
@pytest.mark.parametrize("tokens", [1, 3, 4, 5, 16])
def test_tensor_core_decode_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(11 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, tc_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("m,n,r", [(64, 96, 40), (256, 256, 120)])
@pytest.mark.parametrize("tokens", [1, 7, 16])
def test_tensor_core_decode_integer_bit_exact(P, m, n, r, tokens):
    d = synth.integer_layer(9 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, tc_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


@pytest.mark.parametrize("m,n", [(4096, 4096), (14336, 4096)])
@pytest.mark.parametrize("tokens", [1, 16])
def test_tensor_core_decode_full_size_sampled_rows(P, m, n, tokens):
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(77 + m // 1024 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r, tc_decode=True)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(tokens + 1).choice(m, size=256, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


# n = 1920 and 1792 give 15 and 14 column chunks: with one row block the
# first phase runs clusters of 15 and 14 CTAs, whose slices of 9 and 10 rows
# leave the last CTA 2 rows and no row.
@pytest.mark.parametrize("m,n,r", [(300, 1920, 100), (200, 1792, 90)])
@pytest.mark.parametrize("tokens", [1, 4, 6, 13])
def test_lookup_decode_cluster_slices(P, m, n, r, tokens):
    d = synth.layer_signs(3 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, lut_decode=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    err = O.rowwise_rel_err(y, oracle_from_signs(d, n))
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("tokens", [1, 5, 16])
@pytest.mark.parametrize("kernel", ["default", "tc", "lut", "mma"])
def test_longest_contraction(P, tokens, kernel):
    m, n = 256, 32768
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(5 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r, tc_decode=kernel == "tc", lut_decode=kernel == "lut",
                        mma_decode=kernel == "mma")
    y = run_gpu(layer, d["x"], n)
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r)
    assert O.rowwise_rel_err(y, ref) <= TOL
    layer.free()


def test_unknown_flag_rejected(P):
    import ctypes
    d = synth.layer_signs(53, 64, 96, 20, 1)
    U = torch.from_numpy(d["U"]).cuda()
    V = torch.from_numpy(d["V"]).cuda()
    a, s, b = (torch.from_numpy(d[k].view(np.float16)).cuda() for k in ("a", "s", "b"))
    desc = P._Desc(64, 96, 20, 64 | P.AF1_FLAG_ANY_RANK, 0)
    h = ctypes.c_void_p()
    rc = P._lib.af1_pack_layer(ctypes.byref(desc), U.data_ptr(), V.data_ptr(), a.data_ptr(), s.data_ptr(),
                               b.data_ptr(), None, None, None, ctypes.byref(h))
    assert rc == -1 and not h.value
