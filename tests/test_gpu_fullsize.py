"""Parity at the benchmark's full sizes.

* GPT-2-small shape (12 layers, D=768, vocab 50257, bf16): 8 x 512-token prompts in the
  launch configuration bench.py times (forced exits ~ U{4..12}), then decode steps,
  against the oracle in full; and the threshold mode at delta 0.9.
* Llama-7B shape (32 layers, D=4096, 32 x 128 heads, SwiGLU 11008, vocab 32000, bf16):
  the oracle cannot run the whole model in seconds, so outputs are sampled: the
  skipped-layer fill of 4096 tokens is checked entry by entry for sampled tokens and
  layers against the oracle's projection with weights regenerated on the host, and a
  2048-token prompt pass (exit layers ~ truncated N(24, 4) on [8, 32]) is checked for
  the forced exit layers and, for sampled exited tokens, for the fill property
  cache[r] = layer r's K/V of the token's own mapped state.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from parity_utils import TOL, Pair, assert_rows_close, compare_decode, compare_prefill

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


def test_gpt2_small_bench_configuration_forced_and_decode():
    cfg = synth.gpt2_small_config(max_batch=8, max_seq=520, max_pos=1024)
    pair = Pair(cfg, seed=0)
    B, P = 8, 512
    tokens = synth.make_tokens(0, B, P, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(0, B * P, 4, 12, name="forced_prompt").numpy().reshape(B, P)
    ores, cache, g = compare_prefill(pair, tokens, 0.9, forced)
    fd = synth.forced_exits_uniform(0, 2 * B, 4, 12, name="forced_decode").numpy().reshape(2, B)
    compare_decode(pair, cache, ores.next_token, 2, 0.9, fd)
    pair.compare_cache(cache, B, P + 2)
    pair.close()


def test_gpt2_small_threshold_mode():
    cfg = synth.gpt2_small_config(max_batch=2, max_seq=512, max_pos=1024)
    pair = Pair(cfg, seed=0)
    tokens = synth.make_tokens(1, 2, 256, cfg.vocab).numpy()
    ores, cache, g = compare_prefill(pair, tokens, 0.9)
    compare_decode(pair, cache, ores.next_token, 2, 0.9)
    pair.close()


def _host_layer(cfg, r):
    """Layer r's (1-based) attention-input gain and W_K / W_V, regenerated on the host."""
    shapes = synth.weight_shapes(cfg)
    w = {}
    for n in ("attn_norm.g", "wk", "wv"):
        name = f"layers.{r - 1}.{n}"
        w[name] = synth.make_weight(cfg, name, shapes[name], seed=0)
    return w


def _oracle_kv(cfg, w, r, h, pos):
    """The oracle's K/V projection of layer r for rows h, using only layer r's weights."""
    om = O.OracleModel(cfg, w)
    return om.kv_project(r, h, pos)


@pytest.fixture(scope="module")
def llama7b():
    cfg = synth.llama7b_config(max_batch=4, max_seq=2048, max_pass_tokens=2048, block_shuffle_seed=11)
    W = synth.make_weights(cfg, seed=0, device="cuda")
    m = adept.Model(cfg, W)
    del W
    torch.cuda.empty_cache()
    yield cfg, m
    m.close()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("istar", [4, 24])
def test_llama7b_skipped_layer_fill_sampled(llama7b, istar):
    cfg, m = llama7b
    T, seqs = 4096, 4
    adept.adept_seq_reserve(m.h, [cfg.max_seq] * seqs)
    h = synth.make_mapped_states(5, T, cfg.d_model)
    j = np.arange(T)
    seq, pos = j % seqs, j // seqs
    el = np.full(T, istar)
    dev = lambda x: torch.as_tensor(x, dtype=torch.int32).cuda().contiguous()  # noqa: E731
    adept.adept_skip_kv_fill(m.h, T, h.cuda(), dev(el), dev(seq), dev(pos))
    m.check()
    sample = synth.randint(7, "sample", 16, 0, T - 1).numpy()
    for r in (istar + 1, (istar + 1 + cfg.n_layers) // 2, cfg.n_layers):
        w = _host_layer(cfg, r)
        k, v = _oracle_kv(cfg, w, r, h.double().numpy()[sample], pos[sample])
        for n, t in enumerate(sample):
            gk, gv = m.read_kv(r, int(seq[t]), int(pos[t]), 1)
            assert_rows_close(gk.float().cpu().numpy().reshape(1, -1), k[n].reshape(1, -1), TOL["bf16"], f"K r={r}")
            assert_rows_close(gv.float().cpu().numpy().reshape(1, -1), v[n].reshape(1, -1), TOL["bf16"], f"V r={r}")


def test_llama7b_prompt_pass_forced_exits_and_fill_property(llama7b):
    cfg, m = llama7b
    P = 2048
    tokens = synth.make_tokens(0, 1, P, cfg.vocab).cuda()
    forced = synth.forced_exits_truncnorm(0, P, 24.0, 4.0, 8, 32).view(1, P)
    ex, lg, nx, sim = m.prefill(tokens, 0.9, forced.cuda())
    m.check()
    np.testing.assert_array_equal(ex.cpu().numpy(), forced.numpy().reshape(-1))
    assert torch.isfinite(lg).all()
    final = m.final_states(P).cpu().double().numpy()
    f = forced.numpy().reshape(-1)
    exited = np.nonzero(f < cfg.n_layers)[0]
    sample = exited[synth.randint(9, "sample", 8, 0, len(exited) - 1).numpy()]
    layers = sorted({int(f[sample].max()) + 1, cfg.n_layers})
    for r in layers:
        w = _host_layer(cfg, r)
        rows = [t for t in sample if f[t] < r]
        if not rows:
            continue
        k, v = _oracle_kv(cfg, w, r, final[rows], np.asarray(rows))
        for n, t in enumerate(rows):
            gk, gv = m.read_kv(r, 0, int(t), 1)
            assert_rows_close(gk.float().cpu().numpy().reshape(1, -1), k[n].reshape(1, -1), TOL["bf16"], f"K r={r}")
            assert_rows_close(gv.float().cpu().numpy().reshape(1, -1), v[n].reshape(1, -1), TOL["bf16"], f"V r={r}")
