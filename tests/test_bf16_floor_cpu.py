"""The bf16 noise-floor helper: its rounding is round-to-nearest-even, and with
rounding switched off it is exactly the oracle."""
import numpy as np

import _bf16_floor as fl
import oracle
import synth


def test_bf16_round_is_rne():
    f = synth.normal(9, 1, (50000,), "f32", sigma=3.0)
    h = synth.normal(9, 1, (50000,), "bf16", sigma=3.0)  # generator's own f32 -> bf16 RNE
    assert np.array_equal(fl.bf16_round(f), oracle.widen(h))
    assert fl.bf16_round(np.array([1.0 + 2 ** -8]))[0] == 1.0          # tie -> even
    assert fl.bf16_round(np.array([1.0 + 3 * 2 ** -8]))[0] == 1.0 + 2 ** -6


def test_floor_without_rounding_is_the_oracle(tiny_shape, tiny_weights, monkeypatch):
    toks = synth.tokens((20,), tiny_shape.vocab, stream=3)
    monkeypatch.setattr(fl, "bf16_round", lambda x: np.asarray(x, dtype=np.float64))
    z = fl.forward_logits_bf16_activations(tiny_shape, tiny_weights, toks)
    assert np.abs(z - oracle.forward_logits(tiny_shape, tiny_weights, toks)).max() < 1e-12


def test_floor_with_rounding_is_close_but_not_exact(tiny_shape, tiny_weights):
    toks = synth.tokens((20,), tiny_shape.vocab, stream=3)
    z = oracle.forward_logits(tiny_shape, tiny_weights, toks)
    zf = fl.forward_logits_bf16_activations(tiny_shape, tiny_weights, toks)
    e = np.abs(zf - z).max() / z.std()
    assert 1e-4 < e < 5e-2


def test_decode_rounding_points_without_rounding_are_the_oracle(tiny_shape, tiny_weights, monkeypatch):
    """The decode path's split norm, W (x g s) = s W (x g), is the same function: with
    rounding off, the decode-path floor is the oracle again."""
    toks = synth.tokens((20,), tiny_shape.vocab, stream=3)
    monkeypatch.setattr(fl, "bf16_round", lambda x: np.asarray(x, dtype=np.float64))
    z = fl.forward_logits_bf16_activations(tiny_shape, tiny_weights, toks, decode_from=7)
    assert np.abs(z - oracle.forward_logits(tiny_shape, tiny_weights, toks)).max() < 1e-12


def test_decode_rounding_points_differ_only_after_decode_from(tiny_shape, tiny_weights):
    """Positions before decode_from see the prefill path only (causal); later ones
    are rounded at other points, so they differ from the prefill-path floor."""
    toks = synth.tokens((20,), tiny_shape.vocab, stream=3)
    zp = fl.forward_logits_bf16_activations(tiny_shape, tiny_weights, toks)
    zd = fl.forward_logits_bf16_activations(tiny_shape, tiny_weights, toks, decode_from=12)
    assert np.array_equal(zp[:12], zd[:12])
    assert np.abs(zp[12:] - zd[12:]).max() > 0
    z = oracle.forward_logits(tiny_shape, tiny_weights, toks)
    e = np.abs(zd - z).max() / z.std()
    assert 1e-4 < e < 5e-2
