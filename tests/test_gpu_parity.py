"""CUDA path against the FP64 oracle, through the C ABI.

Bars: packed words bit-exact; integer-exact inputs bit-exact in FP32 output;
everything else within the row-wise infinity-norm relative error of 2e-3.
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


# ---------------------------------------------------------------------------
# Packing
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("m,n,r", [(16, 128, 8), (33, 70, 31), (200, 129, 127), (1000, 1500, 513),
                                   (4096, 4096, 2028)])
def test_pack_words_bit_exact(P, m, n, r):
    d = synth.layer_signs(100 + m, m, n, r, 1)
    layer, Uw, Vw = signs_layer(P, d, return_words=True)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(Uw.cpu().numpy().view(np.uint32), O.pack_U(d["U"]))
    np.testing.assert_array_equal(Vw.cpu().numpy().view(np.uint32), O.pack_V(d["V"]))
    layer.free()


# ---------------------------------------------------------------------------
# Forward vs oracle, small and ragged shapes, all token paths
# ---------------------------------------------------------------------------

SHAPES = [(16, 16, 8), (64, 64, 32), (100, 130, 77), (256, 384, 200), (1000, 700, 321), (520, 2000, 600),
          (1024, 4096, 800)]
TOKENS = [1, 2, 3, 4, 5, 8, 9, 16, 17, 40]


@pytest.mark.parametrize("m,n,r", SHAPES)
@pytest.mark.parametrize("tokens", TOKENS)
def test_forward_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(7 * m + n + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n, torch.float32)
    ref = oracle_from_signs(d, n)
    err = O.rowwise_rel_err(y, ref)
    assert err <= TOL, err
    layer.free()


@pytest.mark.parametrize("m,n,r", [(100, 130, 77), (1000, 700, 321)])
@pytest.mark.parametrize("tokens", [1, 5, 16])
def test_forward_fp16_output(P, m, n, r, tokens):
    d = synth.layer_signs(3 * m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n, torch.float16)
    ref = oracle_from_signs(d, n)
    assert O.rowwise_rel_err(y, ref) <= TOL
    layer.free()


def test_outlier_channels(P):
    """Activations with 1% of channels x20 (the prefill workload's outliers)."""
    m, n, r = 1024, 4096, 800
    d = synth.layer_signs(77, m, n, r, 8, outlier_frac=0.01)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n)
    assert O.rowwise_rel_err(y, oracle_from_signs(d, n)) <= TOL
    layer.free()


# ---------------------------------------------------------------------------
# Exact cases
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (64, 96, 40), (130, 200, 100), (256, 256, 120)])
@pytest.mark.parametrize("tokens", [1, 2, 3, 7, 16])
def test_integer_inputs_bit_exact(P, m, n, r, tokens):
    """Unit scales, x in {-2..2}: every partial sum is an exact small dyadic
    number, so the FP32 output must equal the oracle exactly."""
    d = synth.integer_layer(5 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, any_rank=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    ref = oracle_from_signs(d, n)
    np.testing.assert_array_equal(y, ref)
    layer.free()


def sylvester(k):
    H = np.array([[1]], dtype=np.int8)
    for _ in range(k):
        H = np.block([[H, H], [H, -H]]).astype(np.int8)
    return H


@pytest.mark.parametrize("k", [6, 8])
def test_hadamard_identity(P, k):
    """U = V = H, s = 1/N: the layer is Diag(a * b), so y = a * b * x."""
    N = 2 ** k
    H = sylvester(k)
    g = synth.rng(k)
    a = synth.scales_f16(g, N)
    b = synth.scales_f16(g, N)
    s = np.full(N, np.float16(1.0 / N)).view(np.uint16)
    x = synth.activations_f16(g, 3, N)
    d = dict(U=H, V=H, a=a, s=s, b=b, x=x)
    layer = signs_layer(P, d, any_rank=True)
    y = run_gpu(layer, x, N)
    af, bf, xf = (O.f16_bits_to_f64(v) for v in (a, b, x))
    expect = xf.reshape(3, N) * (af * bf)[None, :]
    assert O.rowwise_rel_err(y, expect) <= TOL
    # integer variant: a = b = 1, integer x -> exact
    one = np.full(N, np.float16(1.0)).view(np.uint16)
    xi = g.integers(-2, 3, size=(2, N)).astype(np.float16).view(np.uint16)
    layer2 = signs_layer(P, dict(U=H, V=H, a=one, s=s, b=one, x=xi), any_rank=True)
    yi = run_gpu(layer2, xi, N)
    np.testing.assert_array_equal(yi, O.f16_bits_to_f64(xi).reshape(2, N))
    layer.free()
    layer2.free()


def test_rank_one_outer_product(P):
    m, n = 300, 500
    d = synth.layer_signs(9, m, n, 1, 4)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n)
    a, s, b = (O.f16_bits_to_f64(d[k]) for k in ("a", "s", "b"))
    W = s[0] * np.outer(a * d["U"][:, 0], b * d["V"][:, 0])
    ref = O.f16_bits_to_f64(d["x"]).reshape(4, n) @ W.T
    assert O.rowwise_rel_err(y, ref) <= TOL
    layer.free()


# ---------------------------------------------------------------------------
# Deployable-format entry point and full-size shapes
# ---------------------------------------------------------------------------

def test_words_entry_matches_signs_entry(P):
    m, n, r = 700, 900, 333
    d = synth.layer_signs(11, m, n, r, 5)
    l1 = signs_layer(P, d)
    dw = dict(Uw=O.pack_U(d["U"]), Vw=O.pack_V(d["V"]), a=d["a"], s=d["s"], b=d["b"])
    l2 = words_layer(P, dw, m, n, r)
    y1 = run_gpu(l1, d["x"], n)
    y2 = run_gpu(l2, d["x"], n)
    assert O.rowwise_rel_err(y1, y2) <= 1e-6
    assert O.rowwise_rel_err(y2, oracle_from_signs(d, n)) <= TOL
    l1.free()
    l2.free()


FULL = [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336), (8192, 8192), (1024, 8192),
        (28672, 8192), (8192, 28672)]


@pytest.mark.parametrize("m,n", FULL)
@pytest.mark.parametrize("tokens", [1, 4, 16])
def test_full_size_sampled_rows(P, m, n, tokens):
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(1000 * m // 1024 + n // 1024 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(tokens).choice(m, size=256, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


FULL_70B = [(8192, 8192), (1024, 8192), (28672, 8192), (8192, 28672)]


@pytest.mark.parametrize("m,n", FULL_70B)
@pytest.mark.parametrize("tokens", [8, 64, 512])
def test_full_size_70b_sampled_rows(P, m, n, tokens):
    """The 70B-class shapes of the decode/prefill crossover sweep at their
    full size: 8 tokens (decode on the 16-bit-operand tensor-core kernel)
    and 64 / 512 tokens (prefill, including the long-K split of the
    8192 x 28672 first GEMM)."""
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(3000 + m // 1024 + n // 1024 + tokens, m, n, r, tokens)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(tokens + 7).choice(m, size=128, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


# ---------------------------------------------------------------------------
# Workspace, streams, graphs and errors
# ---------------------------------------------------------------------------

def test_workspace_shared_across_layers_and_calls(P):
    da = synth.layer_signs(21, 300, 400, 150, 3)
    db = synth.layer_signs(22, 500, 260, 100, 9)
    la, lb = signs_layer(P, da), signs_layer(P, db)
    ws = torch.zeros(max(la.workspace_bytes(16), lb.workspace_bytes(16)), dtype=torch.uint8, device="cuda")
    xa, xb = f16(da["x"]).reshape(3, 400), f16(db["x"]).reshape(9, 260)
    ra, rb = oracle_from_signs(da, 400), oracle_from_signs(db, 260)
    for _ in range(3):
        ya = la.forward(xa, out_dtype=torch.float32, workspace=ws)
        yb = lb.forward(xb, out_dtype=torch.float32, workspace=ws)
        torch.cuda.synchronize()
        assert O.rowwise_rel_err(ya.double().cpu().numpy(), ra) <= TOL
        assert O.rowwise_rel_err(yb.double().cpu().numpy(), rb) <= TOL
    P.workspace_status(ws)
    la.free()
    lb.free()


@pytest.mark.parametrize("tokens", [2, 12])
def test_cuda_graph_replay(P, tokens):
    """A forward call captured in a CUDA graph and replayed: the lookup-table
    kernels (2 tokens) and the 16-bit-operand tensor-core kernel (12)."""
    m, n, r = 1024, 4096, 800
    d = synth.layer_signs(31 + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    x = f16(d["x"]).reshape(tokens, n)
    y = torch.empty((tokens, m), dtype=torch.float32, device="cuda")
    ws = layer.make_workspace()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        layer.forward_into(x, y, ws, stream=s)  # warm-up outside capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        layer.forward_into(x, y, ws, stream=s)
    y.zero_()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert O.rowwise_rel_err(y.double().cpu().numpy(), oracle_from_signs(d, n)) <= TOL
    layer.free()


def test_tokens_zero_is_noop(P):
    d = synth.layer_signs(41, 64, 64, 20, 1)
    layer = signs_layer(P, d)
    x = torch.zeros((0, 64), dtype=torch.float16, device="cuda")
    y = torch.full((1, 64), 7.0, dtype=torch.float32, device="cuda")
    layer.forward_into(x, y, layer.make_workspace())
    torch.cuda.synchronize()
    assert bool((y == 7.0).all())
    layer.free()


def test_error_codes(P):
    d = synth.layer_signs(51, 64, 96, 20, 2)
    layer = signs_layer(P, d)
    ws = layer.make_workspace()
    x = f16(d["x"]).reshape(2, 96)
    y = torch.empty((2, 64), dtype=torch.float16, device="cuda")
    with pytest.raises(P.AF1Error) as e:
        layer.forward_into(x.cpu(), y, ws)
    assert e.value.code == -2
    xbig = torch.zeros((2, 104), dtype=torch.float16, device="cuda")
    with pytest.raises(P.AF1Error) as e:
        layer.forward_into(xbig[:, 1:], y, ws)  # 2-byte offset: misaligned
    assert e.value.code == -3
    with pytest.raises(P.AF1Error) as e:
        layer.forward_into(x, y, ws[:128])
    assert e.value.code == -8
    bad = dict(d)
    bad["U"] = d["U"].copy()
    bad["U"][3, 5] = 0
    with pytest.raises(P.AF1Error) as e:
        signs_layer(P, bad, any_rank=False)
    assert e.value.code == -5
    big = synth.layer_signs(52, 64, 64, 40, 1)
    with pytest.raises(P.AF1Error) as e:
        signs_layer(P, big, any_rank=False)  # r = 40 > 1.0-BPW rank of 64 x 64 (14)
    assert e.value.code == -4
    P.workspace_status(ws)
    layer.free()


def test_first_calls_interleaved_with_other_layers(P):
    """Each layer's first forward call, with a fresh workspace that the
    allocator may place where another layer's workspace just was. Inputs a
    preceding kernel may have written must never be served stale."""
    shapes = [(520, 2000, 600), (1024, 4096, 800), (256, 384, 200), (1024, 4096, 800), (1000, 700, 321)]
    for rep in range(3):
        for i, (m, n, r) in enumerate(shapes):
            tokens = (1, 3, 5, 9, 2)[(i + rep) % 5]
            d = synth.layer_signs(900 + 10 * rep + i, m, n, r, tokens)
            layer = signs_layer(P, d)
            y = run_gpu(layer, d["x"], n, torch.float32)
            ref = oracle_from_signs(d, n)
            for t in range(tokens):
                assert O.rowwise_rel_err(y[t:t + 1], ref[t:t + 1]) <= TOL, (m, n, r, tokens, t)
            layer.free()


# ---------------------------------------------------------------------------
# Prefill path (more than 16 tokens): tcgen05 GEMMs
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (100, 130, 77), (256, 384, 200), (1000, 700, 321),
                                   (1024, 4096, 800)])
@pytest.mark.parametrize("tokens", [17, 128, 129, 300])
def test_prefill_matches_oracle(P, m, n, r, tokens):
    d = synth.layer_signs(31 * m + n + tokens, m, n, r, tokens, outlier_frac=0.01)
    layer = signs_layer(P, d)
    for out_dtype in (torch.float32, torch.float16):
        y = run_gpu(layer, d["x"], n, out_dtype)
        ref = oracle_from_signs(d, n)
        assert O.rowwise_rel_err(y, ref) <= TOL, out_dtype
    layer.free()


@pytest.mark.parametrize("m,n,r", [(64, 96, 40), (130, 200, 100), (256, 256, 120)])
@pytest.mark.parametrize("tokens", [40, 200])
def test_prefill_integer_inputs_bit_exact(P, m, n, r, tokens):
    d = synth.integer_layer(77 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


@pytest.mark.parametrize("m,n", [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336)])
def test_prefill_full_size_sampled_rows(P, m, n):
    """The prefill workload: LLaMA-3-8B-shaped linears, 2048 tokens, 1 % outlier channels x20."""
    tokens = 2048
    r = O.rank_for_budget(m, n, 1)
    d = synth.layer_words(7000 + m // 1024 + n // 1024, m, n, r, tokens, outlier_frac=0.01)
    layer = words_layer(P, d, m, n, r)
    y = run_gpu(layer, d["x"], n)
    rows = np.sort(synth.rng(5).choice(m, size=128, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
    layer.free()


@pytest.mark.parametrize("m,n,r,tokens", [(1024, 8192, 892, 64), (4096, 4096, 2028, 20), (1000, 700, 321, 33)])
def test_prefill_short_pass_split_k(P, m, n, r, tokens):
    """Short passes (few row blocks x token tiles): the persistent grid splits
    K, so tiles are shared by several CTAs and summed from their partials."""
    d = synth.layer_words(8100 + m + tokens, m, n, r, tokens, outlier_frac=0.01)
    layer = words_layer(P, d, m, n, r, any_rank=r > O.rank_for_budget(m, n, 1))
    for out_dtype in (torch.float32, torch.float16):
        y = run_gpu(layer, d["x"], n, out_dtype)
        rows = np.sort(synth.rng(6).choice(m, size=min(m, 128), replace=False))
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
        assert O.rowwise_rel_err(y[:, rows], ref) <= TOL, out_dtype
    layer.free()


# Cases chosen (with the host's grid model) to cover each path of the
# persistent prefill kernel: tiles of 32, 64, 128 and 256 tokens; tiles
# shared by 2, 3, 4 and 8 CTAs, summed in 2-4 pieces of the activation ring;
# two accumulators (tiles of <= 128 tokens) and one (256); both GEMMs
# shared; ragged rows, columns and tokens; whole tiles only.
STREAM_K_CASES = [
    (1024, 8192, 910, 512),   # GEMM 1: 256-token tiles shared by 4 CTAs, 3 ring pieces
    (700, 900, 333, 17),      # GEMM 1: 32-token tiles shared by 3 CTAs, 2 pieces
    (4096, 4096, 2028, 100),  # both GEMMs: 128-token tiles shared by 4 CTAs
    (1024, 4096, 800, 300),   # 256-token tiles shared by 2 CTAs, a ragged second token tile
    (2048, 1536, 700, 64),    # 64-token tiles shared by 3 CTAs
    (384, 5000, 300, 200),    # ragged K (5000), 3 CTAs per tile
    (1024, 8192, 892, 64),    # 64-token tiles shared by 8 CTAs, 4 ring pieces
    (512, 3000, 400, 130),    # whole tiles only
    (3000, 512, 300, 129),    # whole tiles, ragged rows
]


@pytest.mark.parametrize("m,n,r,tokens", STREAM_K_CASES)
def test_prefill_stream_k_paths(P, m, n, r, tokens):
    d = synth.layer_words(8300 + m + n + tokens, m, n, r, tokens, outlier_frac=0.01)
    layer = words_layer(P, d, m, n, r, any_rank=True)
    rows = np.sort(synth.rng(7).choice(m, size=min(m, 160), replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    for out_dtype in (torch.float32, torch.float16):
        y = run_gpu(layer, d["x"], n, out_dtype)
        assert O.rowwise_rel_err(y[:, rows], ref) <= TOL, out_dtype
    layer.free()


@pytest.mark.parametrize("m,n,r,tokens", [(1024, 8192, 910, 512), (700, 900, 333, 17), (4096, 4096, 2028, 100),
                                          (1024, 8192, 892, 64)])
def test_prefill_stream_k_integer_bit_exact_and_deterministic(P, m, n, r, tokens):
    # Shared tiles are summed in contributor order whichever CTA counts last:
    # with integer inputs every partial and sum is exact (bit-for-bit with
    # the oracle), and repeated calls give identical bits.
    d = synth.integer_layer(4242 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, any_rank=True)
    y0 = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y0, oracle_from_signs(d, n))
    for _ in range(2):
        np.testing.assert_array_equal(run_gpu(layer, d["x"], n, torch.float32), y0)
    layer.free()


def test_prefill_two_passes(P):
    """More than 2048 tokens: passes of 2048 (tiles of 256) and a tail pass of
    52 (tiles of 64), the second writing at a token offset."""
    m, n, r, tokens = 1024, 1536, 600, 2100
    d = synth.layer_words(8500, m, n, r, tokens, outlier_frac=0.01)
    layer = words_layer(P, d, m, n, r, any_rank=True)
    rows = np.sort(synth.rng(8).choice(m, size=128, replace=False))
    ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
    for out_dtype in (torch.float32, torch.float16):
        y = run_gpu(layer, d["x"], n, out_dtype)
        assert O.rowwise_rel_err(y[:, rows], ref) <= TOL, out_dtype
    layer.free()


@pytest.mark.parametrize("m,n,r,tokens", [(128, 2048, 128, 64), (256, 1024, 256, 17)])
def test_prefill_split_k_integer_bit_exact(P, m, n, r, tokens):
    # The split-K partials are summed in a fixed order; with integer inputs
    # every partial and sum is exact, so the result matches bit for bit.
    d = synth.integer_layer(91 + m + tokens, m, n, r, tokens)
    layer = signs_layer(P, d, any_rank=True)
    y = run_gpu(layer, d["x"], n, torch.float32)
    np.testing.assert_array_equal(y, oracle_from_signs(d, n))
    layer.free()


def test_prefill_hadamard_identity(P):
    N = 256
    H = sylvester(8)
    g = synth.rng(99)
    a = synth.scales_f16(g, N)
    b = synth.scales_f16(g, N)
    s = np.full(N, np.float16(1.0 / N)).view(np.uint16)
    x = synth.activations_f16(g, 64, N)
    layer = signs_layer(P, dict(U=H, V=H, a=a, s=s, b=b, x=x), any_rank=True)
    y = run_gpu(layer, x, N)
    af, bf, xf = (O.f16_bits_to_f64(v) for v in (a, b, x))
    assert O.rowwise_rel_err(y, xf.reshape(64, N) * (af * bf)[None, :]) <= TOL
    layer.free()
