"""Format variants through the C ABI: BF16 scales, the 2.5-BPW rank, layer
export and layer files."""
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


def bf16_bits(v) -> np.ndarray:
    """float64 values -> BF16 bit patterns, round to nearest even."""
    f = np.asarray(v, dtype=np.float32).view(np.uint32)
    rounded = f + np.uint32(0x7FFF) + ((f >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_tensor(bits) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("m,n,r", [(100, 130, 77), (1000, 700, 321)])
@pytest.mark.parametrize("tokens", [1, 5, 16, 40])
def test_bf16_scales_match_oracle(P, m, n, r, tokens):
    g = synth.rng(m + tokens)
    U, V = synth.signs(g, m, r), synth.signs(g, n, r)
    a, s, b = (bf16_bits(np.abs(g.normal(0, 0.02, k)) + 1e-3) for k in (m, r, n))
    x = synth.activations_f16(g, tokens, n)
    layer = P.Layer.from_signs(torch.from_numpy(U).cuda(), torch.from_numpy(V).cuda(), bf16_tensor(a),
                               bf16_tensor(s), bf16_tensor(b), any_rank=True)
    y = run_gpu(layer, x, n)
    ref = O.forward_from_packed(O.pack_U(U), O.pack_V(V), a, s, b, x, m, n, r, scale_dtype="bf16")
    assert O.rowwise_rel_err(y, ref) <= TOL
    # The layer keeps the exact FP16 values of the BF16 scales.
    _, _, ea, es, eb = layer.export()
    for e, bits in ((ea, a), (es, s), (eb, b)):
        np.testing.assert_array_equal(e.cpu().numpy().astype(np.float64), O.bf16_bits_to_f64(bits))
    layer.free()


# Out of FP16 range (1e5), below its smallest subnormal (1e-30), and a value
# needing a bit below FP16's subnormal resolution 2^-24 (2^-20 (1 + 2^-7)).
@pytest.mark.parametrize("bad", [1e-30, 1e5, 2.0 ** -20 * (1 + 2.0 ** -7)])
def test_bf16_scale_without_fp16_value_rejected(P, bad):
    m, n, r = 16, 32, 8
    g = synth.rng(3)
    U, V = synth.signs(g, m, r), synth.signs(g, n, r)
    a = bf16_bits(np.full(m, 0.5))
    s = bf16_bits(np.full(r, 0.25))
    b = bf16_bits(np.full(n, 0.125))
    b[7] = bf16_bits([bad])[0]
    ok_in_bf16 = O.bf16_bits_to_f64(b[7:8])[0]
    with np.errstate(over="ignore"):
        assert np.float16(ok_in_bf16) != ok_in_bf16 or not np.isfinite(np.float16(ok_in_bf16))
    with pytest.raises(P.AF1Error) as e:
        P.Layer.from_signs(torch.from_numpy(U).cuda(), torch.from_numpy(V).cuda(), bf16_tensor(a),
                           bf16_tensor(s), bf16_tensor(b), any_rank=True)
    assert e.value.code == -1


def test_rank_for_two_and_a_half_bits(P):
    """The paper's 2.5-BPW setting only changes r; the layer runs at that rank."""
    m = n = 4096
    r = P.rank_for_budget(m, n, 5, 2)
    assert r == O.rank_for_budget(m, n, 2.5)
    assert P.storage_bits(m, n, r) <= 2.5 * m * n < P.storage_bits(m, n, r + 1)
    with pytest.raises(P.AF1Error):
        words_layer(P, synth.layer_words(1, m, n, r, 1), m, n, r, any_rank=False)  # above the 1.0-BPW rank
    for tokens in (1, 16):
        d = synth.layer_words(11 + tokens, m, n, r, tokens)
        layer = words_layer(P, d, m, n, r, any_rank=True)
        y = run_gpu(layer, d["x"], n)
        rows = np.sort(synth.rng(tokens).choice(m, size=256, replace=False))
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r, rows=rows)
        assert O.rowwise_rel_err(y[:, rows], ref) <= TOL
        layer.free()


@pytest.mark.parametrize("m,n,r", [(16, 16, 8), (200, 129, 127), (1000, 1500, 513)])
def test_export_matches_oracle_pack(P, m, n, r):
    d = synth.layer_signs(200 + m, m, n, r, 1)
    layer = signs_layer(P, d)
    Uw, Vw, a, s, b = layer.export()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(Uw.cpu().numpy().view(np.uint32), O.pack_U(d["U"]))
    np.testing.assert_array_equal(Vw.cpu().numpy().view(np.uint32), O.pack_V(d["V"]))
    for t, bits in ((a, d["a"]), (s, d["s"]), (b, d["b"])):
        np.testing.assert_array_equal(t.cpu().numpy().view(np.uint16), bits)
    layer.free()


@pytest.mark.parametrize("m,n,r,tokens", [(100, 130, 77, 3), (1024, 4096, 800, 1), (300, 700, 321, 64)])
def test_save_load_round_trip(P, tmp_path, m, n, r, tokens):
    d = synth.layer_signs(300 + m, m, n, r, tokens)
    layer = signs_layer(P, d)
    path = tmp_path / "layer.af1"
    layer.save(path)
    raw = path.read_bytes()
    assert raw[:8] == b"AF1LAYER" and len(raw) == 40 + 4 * (m * O.words_per_row(r) + r * O.words_per_row(n)) + 2 * (m + r + n)
    loaded = P.Layer.load(path)
    assert (loaded.m, loaded.n, loaded.r) == (m, n, r)
    for t1, t2 in zip(layer.export(), loaded.export()):
        assert torch.equal(t1, t2)
    y1 = run_gpu(layer, d["x"], n)
    y2 = run_gpu(loaded, d["x"], n)
    np.testing.assert_array_equal(y1, y2)
    assert O.rowwise_rel_err(y2, oracle_from_signs(d, n)) <= TOL
    layer.free()
    loaded.free()


def test_load_errors(P, tmp_path):
    with pytest.raises(P.AF1Error) as e:
        P.Layer.load(tmp_path / "missing.af1")
    assert e.value.code == -9
    d = synth.layer_signs(7, 16, 32, 8, 1)
    layer = signs_layer(P, d)
    path = tmp_path / "l.af1"
    layer.save(path)
    raw = path.read_bytes()
    (tmp_path / "short.af1").write_bytes(raw[:-2])
    with pytest.raises(P.AF1Error) as e:
        P.Layer.load(tmp_path / "short.af1")
    assert e.value.code == -9
    (tmp_path / "foreign.af1").write_bytes(b"NOTALAYR" + raw[8:])
    with pytest.raises(P.AF1Error) as e:
        P.Layer.load(tmp_path / "foreign.af1")
    assert e.value.code == -9
    layer.free()
