"""The tcgen05 prompt-attention kernel (S and O in tensor memory, P rounded to bf16) against
the oracle and against the mma.sync kernel it replaces.

Shapes reach its paths: head_dim 64 and 128, grouped-query attention, causal decoders and the
bidirectional encoder, prompts of 1 to 3 key tiles with a ragged last tile, and forced exits
that leave tiles of active rows spanning several sequences (rows of different sequences and
positions in one 128-row tile) in deeper layers."""
import numpy as np
import pytest
import torch

import synth
from parity_utils import Pair, compare_prefill, row_rel_err

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


CASES = {
    "gpt2_dh64": dict(family=synth.GPT2, n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ffn=512, vocab=1000,
                      max_pos=512),
    "llama_dh128_gqa": dict(family=synth.LLAMA, n_layers=4, d_model=256, n_heads=4, head_dim=128, n_kv_heads=2,
                            d_ffn=512, vocab=1000),
    "bert_dh64": dict(family=synth.BERT, n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ffn=512, vocab=1000,
                      max_pos=512, n_classes=2),
}


@pytest.mark.parametrize("name", sorted(CASES))
@pytest.mark.parametrize("B,P", [(3, 300), (5, 37)])
def test_tc_attention_prefill_matches_oracle(name, B, P):
    cfg = synth.ModelConfig(dtype="bf16", max_batch=B, max_seq=max(P, 64), hsm_m1=512, hsm_m2=1024,
                            block_shuffle_seed=11, **CASES[name])
    pair = Pair(cfg, seed=70)
    tokens = synth.make_tokens(70, B, P, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(71, B * P, 2, cfg.n_layers).numpy().reshape(B, P)
    compare_prefill(pair, tokens, 0.9, forced)
    pair.close()


@pytest.mark.parametrize("name", sorted(CASES))
def test_tc_attention_equals_mma_kernel_within_rounding(name):
    """The same prompt pass with the tcgen05 kernel and with the mma.sync kernel: exit layers
    equal (forced), final states within the bf16 tolerance of each other."""
    B, P = 4, 200
    cfg = synth.ModelConfig(dtype="bf16", max_batch=B, max_seq=P, hsm_m1=512, hsm_m2=1024, **CASES[name])
    W = synth.make_weights(cfg, seed=72, device="cuda")
    tok = synth.make_tokens(72, B, P, cfg.vocab).cuda()
    fz = synth.forced_exits_uniform(73, B * P, 2, cfg.n_layers).view(B, P).cuda()
    out = []
    for tc in (1, 0):
        m = adept.Model(cfg, W)
        adept.adept_set_option(m.h, adept.OPT_ATTN_TC, tc)
        ex, lg, _, _ = m.prefill(tok, 0.9, fz)
        m.check()
        out.append((ex.cpu().numpy(), m.final_states(B * P).cpu().numpy(), lg.cpu().numpy()))
        m.close()
    np.testing.assert_array_equal(out[0][0], out[1][0])
    assert row_rel_err(out[0][1], out[1][1]).max() < 2e-2
