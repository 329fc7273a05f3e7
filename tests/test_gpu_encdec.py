"""Encoder-decoder models (Sec. 5.2, the OFA setting) on the GPU against the oracle.

An encoder with token-level exits runs its prompt pass; its final states (s_N, or s~_N of
exited tokens) become, through adept_set_cross_source, the source of every decoder layer's
cross-attention (ragged source lengths per sequence); the decoder runs its own early-exit
prompt pass and greedy generation steps (graph-replayed from the second step on).  Each
side uses its own encoder states, so the comparison is end to end: encoder final states
and classifier logits, decoder exit layers, similarities, final states, logits, greedy
tokens and every cached self-attention K/V entry.  fp32 at a tiny shape (forced exits and
threshold mode) and bf16 at the OFA-base shape (6 + 6 layers, D 768, 12 heads, FFN 3072)."""
import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from parity_utils import Pair, compare_decode, compare_prefill

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


def _tiny(dtype="f32"):
    enc = synth.ModelConfig(family=synth.BERT, n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ffn=1024,
                            vocab=1000, max_pos=64, n_classes=3, dtype=dtype, max_batch=3, max_seq=40)
    dec = synth.ModelConfig(family=synth.GPT2, n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ffn=1024,
                            vocab=1000, max_pos=64, dtype=dtype, max_batch=3, max_seq=48, max_src=40)
    return enc, dec


def _run(enc, dec, seed, src_lens, tgt_len, steps, enc_forced, dec_forced, delta_dec=0.0, std=0.02):
    B, S = len(src_lens), enc.max_seq
    pe = Pair(enc, seed=seed, std=std)
    pd = Pair(dec, seed=seed + 1, std=std)
    src = synth.make_tokens(seed, B, S, enc.vocab).numpy()
    oe, _, ge = compare_prefill(pe, src, 0.9, enc_forced)
    o_states = [oe.final.reshape(B, S, -1)[b, :src_lens[b]] for b in range(B)]
    g_fin = pe.gm.final_states(B * S).view(B, S, -1)
    g_states = torch.cat([g_fin[b, :src_lens[b]] for b in range(B)]).contiguous()
    pd.cross = O.CrossSource(pd.om, o_states)
    pd.gm.set_cross_source(src_lens, g_states)
    tgt = synth.make_tokens(seed + 2, B, tgt_len, dec.vocab).numpy()
    od, cache, _ = compare_prefill(pd, tgt, delta_dec, dec_forced)
    fs = None
    if dec_forced is not None:
        fs = synth.forced_exits_uniform(seed + 3, steps * B, 2, dec.n_layers, name="forced_decode").numpy()
        fs = fs.reshape(steps, B)
    compare_decode(pd, cache, od.next_token, steps, delta_dec, fs)
    pd.compare_cache(cache, B, tgt_len + steps)
    pe.close()
    pd.close()
    return od


def test_encdec_fp32_forced_exits_ragged_sources():
    enc, dec = _tiny()
    B, S = 3, enc.max_seq
    ef = synth.forced_exits_uniform(60, B * S, 2, enc.n_layers).numpy().reshape(B, S)
    df = synth.forced_exits_uniform(61, B * 20, 2, dec.n_layers).numpy().reshape(B, 20)
    _run(enc, dec, 60, [40, 33, 17], 20, 3, ef, df)


def test_encdec_fp32_threshold_decoder():
    enc, dec = _tiny()
    B, S = 3, enc.max_seq
    ef = synth.forced_exits_uniform(62, B * S, 2, enc.n_layers).numpy().reshape(B, S)
    # a threshold inside the decoder's similarity range, so that some tokens leave early
    od = _run(enc, dec, 62, [40, 21, 9], 16, 3, ef, None, delta_dec=0.6, std=0.05)
    assert od.exit_layer.min() >= 2


def test_encdec_bf16_ofa_base_shape():
    enc, dec = synth.ofa_base_configs(src_len=128, tgt_len=24, batch=4)
    B, S = 4, enc.max_seq
    ef = synth.forced_exits_uniform(64, B * S, 2, enc.n_layers).numpy().reshape(B, S)
    df = synth.forced_exits_uniform(65, B * 16, 2, dec.n_layers).numpy().reshape(B, 16)
    _run(enc, dec, 64, [128, 97, 64, 33], 16, 4, ef, df)


def test_encdec_needs_its_source():
    enc, dec = _tiny()
    m = adept.Model(dec, synth.make_weights(dec, seed=66))
    tk = torch.zeros(1, 4, dtype=torch.int32, device="cuda")
    with pytest.raises(adept.AdeptError) as ei:
        m.prefill(tk, 0.9)
    assert ei.value.status == 1
    with pytest.raises(adept.AdeptError):
        m.set_cross_source([enc.max_seq + 1], torch.zeros(enc.max_seq + 1, dec.d_model, device="cuda"))
    m.close()
    me = adept.Model(enc, synth.make_weights(enc, seed=67))
    with pytest.raises(adept.AdeptError):   # an encoder has no cross-attention
        me.set_cross_source([4], torch.zeros(4, enc.d_model, device="cuda"))
    me.close()
