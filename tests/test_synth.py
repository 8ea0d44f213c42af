"""The shared input generators: determinism, padding and distributions."""
import numpy as np

import synth
from oracle import af1_oracle as O


def test_layer_words_padding_and_determinism():
    d1 = synth.layer_words(5, 100, 200, 77, 2)
    d2 = synth.layer_words(5, 100, 200, 77, 2)
    for k in d1:
        np.testing.assert_array_equal(d1[k], d2[k])
    assert d1["Uw"].shape == (100, 4) and d1["Vw"].shape == (77, 8)
    assert O.padding_is_zero(d1["Uw"], 77)
    assert O.padding_is_zero(d1["Vw"], 200)


def test_layer_words_bits_are_balanced():
    d = synth.layer_words(1, 512, 512, 256, 1)
    U = O.unpack_U(d["Uw"], 256)
    assert abs(U.mean()) < 0.01


def test_scales_distribution():
    g = synth.rng(0)
    v = synth.scales_f16(g, 100000).view(np.float16).astype(np.float64)
    assert v.min() >= 1e-3 * (1 - 1e-3)
    # E|N(0, 0.02)| = 0.02 * sqrt(2 / pi)
    assert abs(v.mean() - (0.02 * np.sqrt(2 / np.pi) + 1e-3)) < 5e-4


def test_outlier_channels():
    g = synth.rng(3)
    x = synth.activations_f16(g, 64, 1000, outlier_frac=0.01).view(np.float16).astype(np.float64)
    col_rms = np.sqrt((x ** 2).mean(axis=0))
    assert (col_rms > 8).sum() == 10
