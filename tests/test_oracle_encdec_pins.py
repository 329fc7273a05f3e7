"""Pins of the oracle's encoder-decoder pass (Sec. 5.2, the OFA setting) against the
independent torch reference (no GPU).

The encoder runs its own early-exit pass; its final states (s_N, or s~_N of exited tokens)
are the source of every decoder layer's cross-attention; the decoder runs the early-exit
pass with its own mapper and skipped-layer K/V.  Pinned here:

* delta = +inf everywhere reduces the pair to a plain encoder-decoder forward (batched SDPA,
  ragged sources), prompt pass and cached generation steps;
* forced exits in the decoder (every assignment in {2, 3}^5 on three layers) equal a
  one-token-at-a-time unfold that cross-attends to the encoder's early-exit states;
* the bf16 contract of the cross-attention (encoder states rounded before the K/V
  projection, Q and the source K/V rounded, the attention output rounded before W_Oc)
  equals torch's own bf16 casts, and dropping any one rounding point moves it.
"""
import itertools

import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from torch_reference import TorchRef


def _pair_cfgs(dtype="f32", n_enc=3, n_dec=3, D=16, heads=2, dh=8, src=7, tgt=8):
    enc = synth.ModelConfig(family=synth.BERT, n_layers=n_enc, d_model=D, n_heads=heads, head_dim=dh, d_ffn=2 * D,
                            vocab=40, max_pos=32, n_classes=3, dtype=dtype, max_batch=3, max_seq=src)
    dec = synth.ModelConfig(family=synth.GPT2, n_layers=n_dec, d_model=D, n_heads=heads, head_dim=dh, d_ffn=2 * D,
                            vocab=37, max_pos=32, dtype=dtype, max_batch=3, max_seq=tgt, max_src=src)
    return enc, dec


def _models(enc, dec, seed, std=0.3):
    We = synth.make_weights(enc, seed=seed, std=std, gain_std=0.1)
    Wd = synth.make_weights(dec, seed=seed + 1, std=std, gain_std=0.1)
    return O.OracleModel(enc, We), O.OracleModel(dec, Wd), TorchRef(enc, We, dec.dtype == "bf16"), \
        TorchRef(dec, Wd, dec.dtype == "bf16")


def _encode(me, enc, src_tokens, delta, forced=None):
    B, S = src_tokens.shape
    r = O.prefill(me, O.OracleCache(enc, B, S), src_tokens, delta, forced)
    return r, r.final.reshape(B, S, -1)


def test_cross_weights_exist_only_for_cross_attention_decoders():
    enc, dec = _pair_cfgs()
    names = synth.weight_shapes(dec)
    assert names["layers.0.cwq"] == (dec.d_q, dec.d_model) and names["layers.2.cbo"] == (dec.d_model,)
    assert not any("cw" in k for k in synth.weight_shapes(enc))
    plain = synth.ModelConfig(**{**dec.__dict__, "max_src": 0})
    assert not any(".cw" in k or "cross_norm" in k for k in synth.weight_shapes(plain))
    md = O.OracleModel(dec, synth.make_weights(dec, seed=1))
    with pytest.raises(ValueError):
        O.prefill(md, O.OracleCache(dec, 1, 8), np.zeros((1, 3), dtype=np.int64), np.inf)


def test_full_depth_encoder_decoder_matches_standard_model():
    """delta = +inf in both stacks: the oracle's prompt pass and cached generation steps equal
    a plain batched encoder-decoder forward (SDPA) of the longer target, with a ragged source
    (the second sequence sees only its first 5 source states)."""
    enc, dec = _pair_cfgs()
    me, md, re_, rd = _models(enc, dec, seed=30)
    src = synth.make_tokens(30, 2, 7, enc.vocab).numpy()
    _, E = _encode(me, enc, src, np.inf)
    want_e = re_.full_forward(torch.as_tensor(src)).numpy()
    np.testing.assert_allclose(E, want_e, rtol=1e-10, atol=1e-10)
    states = [E[0], E[1, :5]]
    cs = O.CrossSource(md, states)
    np.testing.assert_array_equal(cs.src_len, [7, 5])
    tgt = synth.make_tokens(31, 2, 8, dec.vocab).numpy()
    cache = O.OracleCache(dec, 2, 8)
    r = O.prefill(md, cache, tgt[:, :5], np.inf, cross=cs)
    ref_src = [torch.as_tensor(s) for s in states]
    want = rd.full_forward(torch.as_tensor(tgt[:, :5]), source=ref_src).numpy()
    np.testing.assert_allclose(r.final.reshape(want.shape), want, rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(r.logits, rd.head(torch.as_tensor(want[:, -1])).numpy(), rtol=1e-10, atol=1e-10)
    for t in range(5, 8):
        r = O.decode_step(md, cache, tgt[:, t], np.inf, cross=cs)
        want = rd.full_forward(torch.as_tensor(tgt[:, :t + 1]), source=ref_src).numpy()[:, -1]
        np.testing.assert_allclose(r.final, want, rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(r.logits, rd.head(torch.as_tensor(want)).numpy(), rtol=1e-10, atol=1e-10)


def test_source_length_and_content_matter():
    """The cross-attention is not a no-op: changing one source state or shortening the
    source changes the decoder's final states."""
    enc, dec = _pair_cfgs()
    me, md, _, _ = _models(enc, dec, seed=32)
    _, E = _encode(me, enc, synth.make_tokens(32, 1, 7, enc.vocab).numpy(), np.inf)
    tgt = synth.make_tokens(33, 1, 4, dec.vocab).numpy()
    base = O.prefill(md, O.OracleCache(dec, 1, 8), tgt, np.inf, cross=O.CrossSource(md, [E[0]])).final
    E2 = E[0].copy()
    E2[3] += 1.0
    moved = O.prefill(md, O.OracleCache(dec, 1, 8), tgt, np.inf, cross=O.CrossSource(md, [E2])).final
    short = O.prefill(md, O.OracleCache(dec, 1, 8), tgt, np.inf, cross=O.CrossSource(md, [E[0, :6]])).final
    assert np.max(np.abs(moved - base)) > 1e-4 and np.max(np.abs(short - base)) > 1e-4


def test_decoder_forced_exits_equal_token_major_unfold_over_an_early_exit_encoder():
    """Encoder tokens leave at forced layers (their s~_N become source states); every decoder
    assignment in {2, 3}^5 (three layers): the layer-major parallel pass equals the
    one-token-at-a-time unfold of the torch reference in exit layers, final states and every
    cached self-attention K/V entry."""
    enc, dec = _pair_cfgs(n_enc=4, n_dec=3, D=8, heads=2, dh=4, src=6, tgt=8)
    me, md, _, rd = _models(enc, dec, seed=34, std=0.4)
    src = synth.make_tokens(34, 1, 6, enc.vocab).numpy()
    re_enc, E = _encode(me, enc, src, 0.0, np.array([2, 3, 4, 2, 3, 4]))
    np.testing.assert_array_equal(re_enc.exit_layer, [2, 3, 4, 2, 3, 4])
    cs = O.CrossSource(md, [E[0]])
    tgt = synth.make_tokens(35, 1, 5, dec.vocab).numpy()
    for assign in itertools.product([2, 3], repeat=5):
        forced = np.array(assign)
        cache = O.OracleCache(dec, 1, 8)
        r = O.prefill(md, cache, tgt, 0.5, forced, cross=cs)
        fin, el, K, V = rd.token_major(tgt[0], forced, source=torch.as_tensor(E[0]))
        np.testing.assert_array_equal(r.exit_layer, el.numpy())
        np.testing.assert_allclose(r.final, fin.numpy(), rtol=1e-11, atol=1e-12)
        for i in range(1, 4):
            for j in range(5):
                np.testing.assert_allclose(cache.K[i - 1][0, j], K[i][j].numpy(), rtol=1e-11, atol=1e-12)
                np.testing.assert_allclose(cache.V[i - 1][0, j], V[i][j].numpy(), rtol=1e-11, atol=1e-12)


def _bf16_cross_gap(md, rd, tgt, forced, E):
    rel = lambda a, b: float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))  # noqa: E731
    cache = O.OracleCache(md.cfg, 1, 8)
    r = O.prefill(md, cache, tgt, 0.5, forced, cross=O.CrossSource(md, [E]))
    fin, el, K, V = rd.token_major(tgt[0], forced, source=torch.as_tensor(E))
    np.testing.assert_array_equal(r.exit_layer, el.numpy())
    gaps = [rel(r.final, fin.numpy()), rel(r.logits, rd.head(fin[-1:]).numpy())]
    for i in range(1, md.cfg.n_layers + 1):
        for j in range(tgt.shape[1]):
            gaps.append(rel(cache.K[i - 1][0, j], K[i][j].numpy()))
            gaps.append(rel(cache.V[i - 1][0, j], V[i][j].numpy()))
    return max(gaps)


def test_bf16_cross_attention_contract_matches_independent_statement(monkeypatch):
    """bf16 decoder with cross-attention and forced exits: the oracle equals the reference's
    bf16 statement to ~1e-12; dropping any single rounding point of the oracle (each call of
    OracleModel.rb in turn, including the cross-attention's) moves it by more than 1e-6."""
    enc, dec = _pair_cfgs(dtype="bf16", n_dec=4, D=32, heads=2, dh=16, src=7)
    Wd = synth.make_weights(dec, seed=36, std=0.2, gain_std=0.1)
    md, rd = O.OracleModel(dec, Wd), TorchRef(dec, Wd, bf16=True)
    E = synth.normal(36, "source_states", (7, dec.d_model), dtype=torch.float64).numpy()
    tgt = synth.make_tokens(37, 1, 6, dec.vocab).numpy()
    forced = np.array([2, 4, 3, 2, 4, 3])
    assert _bf16_cross_gap(md, rd, tgt, forced, E) < 1e-12
    rb = O.OracleModel.rb
    calls = {"n": 0, "skip": -1}

    def counting_rb(self, x):
        calls["n"] += 1
        return x if calls["n"] - 1 == calls["skip"] else rb(self, x)

    monkeypatch.setattr(O.OracleModel, "rb", counting_rb)
    _bf16_cross_gap(md, rd, tgt, forced, E)
    total = calls["n"]
    assert total >= 13 * dec.n_layers   # includes the cross-attention's points
    for k in range(total):
        calls["n"], calls["skip"] = 0, k
        assert _bf16_cross_gap(md, rd, tgt, forced, E) > 1e-6, f"rounding point {k} of {total} has no effect"
