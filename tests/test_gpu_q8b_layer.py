"""GPU parity on one Qwen3-8B-shaped layer (H 4096, 32/8 heads, d 128, I 12288,
bf16): a decode step at batch 1, 8, 16, 32, 64 over a KV cache of 2048 N(0,1) bf16
entries, new token at position 2048.  Compared: the layer's residual output and
the key/value written at position 2048, max |error| <= 3e-2 x std."""
import numpy as np
import pytest

import oracle
import synth
from _gpu import assert_logits_close, decoder

pytestmark = pytest.mark.gpu
S = 2048


@pytest.fixture(scope="module")
def layer_model():
    s = synth.shape("q8b_layer", vocab=1024)
    dec, W = decoder(s, synth.LazyWeights(s))
    return s, dec, oracle.layer_weights(W, 0)


@pytest.mark.parametrize("B", [1, 8, 16, 32, 64])
def test_one_layer_decode_step(layer_model, B):
    import torch
    s, dec, Lw = layer_model
    kc, vc = synth.kv_fill(B, s.n_kv_heads, S, s.head_dim)
    x = synth.hidden_input(B, s.hidden)
    kv = dec.new_kv(B, S + 1)
    view = dec.kv_view(kv, B, S + 1)
    view[0, 0, :, :, :S] = torch.from_numpy(kc.view(np.int16)).view(torch.bfloat16).cuda()
    view[0, 1, :, :, :S] = torch.from_numpy(vc.view(np.int16)).view(torch.bfloat16).cuda()
    xd = torch.from_numpy(x).cuda()
    pos = torch.full((B,), S, dtype=torch.int32, device="cuda")
    dec.decode_layer(0, kv, B, S + 1, xd, pos)
    assert dec.check_status() == 0
    out, kn, vn = oracle.layer_decode_step(s, Lw, x, kc, vc, [S] * B)
    assert_logits_close(xd.cpu().numpy(), out, 3e-2)
    k_gpu = view[0, 0, :, :, S].float().cpu().numpy()
    v_gpu = view[0, 1, :, :, S].float().cpu().numpy()
    assert_logits_close(k_gpu, kn, 3e-2)
    assert_logits_close(v_gpu, vn, 3e-2)
    # the cache entries before position 2048 are untouched
    assert torch.equal(view[0, 0, :, :, :S].cpu(), torch.from_numpy(kc.view(np.int16)).view(torch.bfloat16))


def test_one_layer_decode_ragged_positions_nan_tail(layer_model):
    """Rows at positions 0, 1, 63, 64, 65, 1000, 4095, 8191 in one step; cache memory past
    each row's position is NaN, which must not leak into the output (masked keys, zeroed V)."""
    import torch
    s, dec, Lw = layer_model
    pos = [0, 1, 63, 64, 65, 1000, 4095, 8191]
    B, S = len(pos), 8192
    kc, vc = synth.kv_fill(B, s.n_kv_heads, S, s.head_dim)
    x = synth.hidden_input(B, s.hidden)
    kv = dec.new_kv(B, S)
    view = dec.kv_view(kv, B, S)
    view[0, 0] = torch.from_numpy(kc.view(np.int16)).view(torch.bfloat16).cuda()
    view[0, 1] = torch.from_numpy(vc.view(np.int16)).view(torch.bfloat16).cuda()
    for b, p in enumerate(pos):
        view[0, :, b, :, p:] = float("nan")
    xd = torch.from_numpy(x).cuda()
    dec.decode_layer(0, kv, B, S, xd, torch.tensor(pos, dtype=torch.int32, device="cuda"))
    assert dec.check_status() == 0
    out, kn, vn = oracle.layer_decode_step(s, Lw, x, kc, vc, pos)
    got = xd.cpu().numpy()
    assert np.all(np.isfinite(got))
    assert_logits_close(got, out, 3e-2)
    for b, p in enumerate(pos):
        assert_logits_close(view[0, 0, b, :, p].float().cpu().numpy(), kn[b], 3e-2)
