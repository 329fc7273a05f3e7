"""Element-wise parity with the oracle at the real layer shapes of the two large workloads.

* Llama-2-7B layer shapes (D = 4096, 32 heads x 128, SwiGLU 11008, vocabulary 32000, the
  36 D^2 mapper with widths 8192 / 32768, bf16) with 5 layers instead of 32, so that the
  oracle finishes in seconds: a 256-token prompt pass with forced exits drawn from the
  benchmark's truncated normal scaled to 5 layers (mean 3.75, sd 0.625 on [2, 5]), then 4
  generation steps (batch 1: the weight-streaming GEMM's persistent grid at K = 4096,
  N = 12288 / 22016, and the captured step graph from the second step on), and a threshold
  run whose delta is the median of the layer-2 similarities.  Final states, logits, greedy
  tokens, similarities (the decision rule outside the band) and every cached K/V entry of
  every layer are compared.
* BERT-base at full size (12 layers, D = 768, 64 x 128 tokens, bidirectional): forced exits
  ~ U{4..12} (the benchmark's law) and a threshold run at the median layer-2 similarity;
  final states, classifier logits and every cached K/V entry.

Layer i (1-based) of the paper's pass, Sec. 4.1 exit rule, Sec. 4.2 mapper, Sec. 4.3 KV
generation, App. I dynamic shrinkage.
"""
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


def _median_layer2_similarity(pair, tokens, forced):
    """delta for a threshold run: the median of the oracle's layer-2 similarities (every
    token is tested there), rounded to 1e-3."""
    cfg = pair.cfg
    cache = O.OracleCache(cfg, cfg.max_batch, cfg.max_seq)
    r = O.prefill(pair.om, cache, tokens, 0.0, forced)
    return float(np.round(np.median(r.sim[:, 1]), 3))


@pytest.fixture(scope="module")
def llama_layers():
    cfg = synth.llama7b_config(n_layers=5, max_batch=1, max_seq=264, max_pass_tokens=256, block_shuffle_seed=5)
    W = synth.make_weights(cfg, seed=0, device="cuda")
    pair = Pair(cfg, weights=W)
    del W
    torch.cuda.empty_cache()
    yield pair
    pair.close()
    torch.cuda.empty_cache()


def test_llama7b_layer_shapes_forced_prefill_and_decode(llama_layers):
    pair = llama_layers
    cfg = pair.cfg
    P = 256
    tokens = synth.make_tokens(0, 1, P, cfg.vocab).numpy()
    forced = synth.forced_exits_truncnorm(0, P, 3.75, 0.625, 2, cfg.n_layers).numpy().reshape(1, P)
    assert len(np.unique(forced)) == cfg.n_layers - 1     # exits at every eligible layer and full depth
    ores, cache, g = compare_prefill(pair, tokens, 0.9, forced)
    fd = synth.forced_exits_truncnorm(1, 4, 3.75, 0.625, 2, cfg.n_layers, name="forced_decode").numpy().reshape(4, 1)
    compare_decode(pair, cache, ores.next_token, 4, 0.9, fd)
    pair.compare_cache(cache, 1, P + 4)


def test_llama7b_layer_shapes_threshold(llama_layers):
    pair = llama_layers
    cfg = pair.cfg
    P = 256
    tokens = synth.make_tokens(2, 1, P, cfg.vocab).numpy()
    forced = np.full((1, P), cfg.n_layers)
    delta = _median_layer2_similarity(pair, tokens, forced)
    ores, cache, g = compare_prefill(pair, tokens, delta)
    depth = ores.exit_layer
    assert (depth == 2).any() and (depth > 2).any(), "the threshold run should mix exit depths"
    compare_decode(pair, cache, ores.next_token, 2, delta)
    pair.compare_cache(cache, 1, P + 2)


@pytest.fixture(scope="module")
def llama_layers_b3():
    cfg = synth.llama7b_config(n_layers=5, max_batch=3, max_seq=24, max_pass_tokens=48, block_shuffle_seed=6)
    W = synth.make_weights(cfg, seed=3, device="cuda")
    pair = Pair(cfg, weights=W)
    del W
    torch.cuda.empty_cache()
    yield pair
    pair.close()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("fused_exit", [1, 0])
def test_llama7b_layer_shapes_three_sequences_exit_step(llama_layers_b3, fused_exit):
    """Three sequences per generation step at the Llama-7B layer shapes, forced exits that differ
    between the sequences of a step (every step keeps some rows and drops others at each layer),
    then a threshold step: with the exit step inside the next layer's QKV launch (several rows
    reduced and compacted by every CTA, records written by one) and with the separate exit
    kernel, each against the oracle; every cached K/V entry at the end."""
    pair = llama_layers_b3
    cfg = pair.cfg
    adept.adept_set_option(pair.gm.h, adept.OPT_FUSED_EXIT, fused_exit)
    try:
        B, P = 3, 12
        tokens = synth.make_tokens(10 + fused_exit, B, P, cfg.vocab).numpy()
        forced = synth.forced_exits_uniform(10, B * P, 2, cfg.n_layers).numpy().reshape(B, P)
        ores, cache, g = compare_prefill(pair, tokens, 0.9, forced)
        fd = np.array([[2, 4, 5], [5, 3, 2], [3, 5, 4], [4, 2, 3]])
        compare_decode(pair, cache, ores.next_token, 4, 0.9, fd)
        compare_decode(pair, cache, ores.next_token, 1, 0.9995)
        pair.compare_cache(cache, B, P + 5)
    finally:
        adept.adept_set_option(pair.gm.h, adept.OPT_FUSED_EXIT, 1)


@pytest.fixture(scope="module")
def bert_base():
    cfg = synth.bert_base_config(max_batch=64, max_seq=128, max_pass_tokens=64 * 128)
    W = synth.make_weights(cfg, seed=0, device="cuda")
    pair = Pair(cfg, weights=W)
    del W
    torch.cuda.empty_cache()
    yield pair
    pair.close()
    torch.cuda.empty_cache()


def test_bert_base_full_size_forced(bert_base):
    pair = bert_base
    B, P = 64, 128
    tokens = synth.make_tokens(0, B, P, pair.cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(0, B * P, 4, 12, name="forced_encoder").numpy().reshape(B, P)
    compare_prefill(pair, tokens, 0.9, forced)


def test_bert_base_full_size_threshold(bert_base):
    pair = bert_base
    B, P = 64, 128
    tokens = synth.make_tokens(1, B, P, pair.cfg.vocab).numpy()
    delta = _median_layer2_similarity(pair, tokens, np.full((B, P), pair.cfg.n_layers))
    ores, _, _ = compare_prefill(pair, tokens, delta)
    assert (ores.exit_layer == 2).any() and (ores.exit_layer > 2).any()
