"""Host logic of bench.py's algorithmic-work accounting (the numerators of every roofline and
TFLOP/s figure), pinned to the per-token costs that follow from the model shapes by hand:
a GPT-2-small layer 2 * 12 * 768^2 = 14.16 MFLOP per token, the Table S1 mapper 2 * 72 * D^2
(84.9 MFLOP at D = 768), a Llama-2-7B layer 404.75 MFLOP, its 36 D^2 mapper 1.21 GFLOP and
its K/V projection 2 * D * 2 * D_kv = 67.1 MFLOP per token and layer."""
import numpy as np
import pytest

import bench
import synth


def test_gemm_work_closed_form():
    assert bench.gemm_work(3, 5, 7) == (2.0 * 3 * 5 * 7, float(5 * 7 * 2 + 3 * 7 * 2))
    assert bench.gemm_work(0, 5, 7) == (0.0, 0.0)


def gpt2():
    return synth.gpt2_small_config(max_batch=8, max_seq=640)


def llama():
    return synth.llama7b_config(max_batch=1, max_seq=2304)


def test_gpt2_full_depth_prompt_pass():
    """All tokens at full depth: T layers of 14.16 MFLOP each token plus one head row per
    sequence; no mapper, no fill."""
    c = gpt2()
    T, n_seq = 96, 3
    fl, _ = bench.pass_work(c, np.full(T, c.n_layers), decode=False, n_seq=n_seq)
    layer = 2 * 12 * 768 ** 2
    assert abs(layer - 14.156e6) < 1e3
    assert fl == pytest.approx(T * c.n_layers * layer + 2.0 * n_seq * c.vocab * 768, rel=1e-12)


def test_gpt2_mapper_cost_per_exit():
    """The mapper term: hsm=True minus hsm=False is 2 * 72 * D^2 per exiting token (Table S1,
    84.9 MFLOP at D = 768, about six layers)."""
    c = gpt2()
    e = np.array([4, 4, 7, 12, 12, 9])
    a = bench.pass_work(c, e, decode=False, n_seq=1)[0]
    b = bench.pass_work(c, e, decode=False, n_seq=1, hsm=False)[0]
    exits = int(np.sum(e < c.n_layers))
    assert (a - b) == pytest.approx(exits * 2 * 72 * 768 ** 2, rel=1e-12)
    assert 2 * 72 * 768 ** 2 == pytest.approx(84.9e6, rel=1e-3)


def test_gpt2_prompt_fill_terms():
    """A token leaving at layer i has its K/V projected at every later layer r >= i + 1 of the
    prompt pass (counted from layer 3 on, the first layer after the first eligible exit)."""
    c = gpt2()
    e = np.array([4])
    full = bench.pass_work(c, np.array([c.n_layers]), decode=False, n_seq=1, hsm=False)[0]
    ex = bench.pass_work(c, e, decode=False, n_seq=1, hsm=False)[0]
    layer = 2 * 12 * 768 ** 2
    kv = 2.0 * 2 * 768 * 768
    assert full - ex == pytest.approx((c.n_layers - 4) * (layer - kv), rel=1e-12)


def test_llama_layer_mapper_and_fill_costs():
    c = llama()
    D, F = 4096, 11008
    layer = 2 * (D * 3 * D + D * D + 2 * F * D + F * D)
    assert layer == pytest.approx(404.75e6, rel=1e-4)
    assert 2 * 36 * D ** 2 == pytest.approx(1.208e9, rel=1e-3)
    one = bench.pass_work(c, np.array([c.n_layers]), decode=True, hsm=False)[0]
    assert one == pytest.approx(c.n_layers * layer + 2.0 * c.vocab * D, rel=1e-12)
    fl, _ = bench.decode_fill_work(c, np.array([24]))
    assert fl == pytest.approx((c.n_layers - 24) * 2 * D * 2 * D, rel=1e-12)
    assert 2 * D * 2 * D == pytest.approx(67.1e6, rel=1e-3)


def test_llama_work_identity_mapper_and_head_rows():
    """llama_work: one head row for the one-sequence prompt pass; hsm=False drops exactly the
    mapper's 2 * 36 D^2 per exiting token (prompt and generation steps)."""
    c = llama()
    ep = np.array([24, 32, 20, 32])
    ed = np.array([[30], [32], [12]])
    a = bench.llama_work(c, ep, ed)
    b = bench.llama_work(c, ep, ed, hsm=False)
    exits = int(np.sum(ep < 32) + np.sum(ed < 32))
    assert a - b == pytest.approx(exits * 2 * 36 * 4096 ** 2, rel=1e-12)
    full = bench.llama_work(c, np.full(4, 32), np.full((3, 1), 32))
    per = 2 * (4096 * 3 * 4096 + 4096 * 4096 + 2 * 11008 * 4096 + 11008 * 4096)
    assert full == pytest.approx(7 * 32 * per + 4 * 2.0 * c.vocab * 4096, rel=1e-12)


def test_hsm_train_flops():
    """Training products: 6 x the mapper's weights per example, plus the head forward and input
    gradient (decoders, 4 D V) or the pooler forward and input gradient on the labelled rows
    (encoders, 4 D^2 each)."""
    g = gpt2()
    fc = 2 * 768 * 3072 + 2 * 3072 * 6144
    assert bench.hsm_train_flops(g, 10) == pytest.approx(10 * (6.0 * fc + 4.0 * 768 * g.vocab), rel=1e-12)
    e = synth.bert_base_config()
    assert bench.hsm_train_flops(e, 10, 2) == pytest.approx(10 * 6.0 * fc + 2 * 4.0 * 768 ** 2, rel=1e-12)


def test_fill_micro_work_counts_the_oracles_fill():
    """The fill grid's numerators (bench.fill_micro_work) against a count over what the oracle's
    skipped-layer fill computes (Sec. 4.3) on a small Llama-shaped model with the grid's law (all
    T tokens leaving at i*): every produced (token, layer) entry is two products of the layer's
    K and V weight shapes; each filled layer's W_K / W_V is read once, each s~ once, each entry
    written once (bf16 throughout)."""
    from oracle import adept_oracle as O
    cfg = synth.ModelConfig(family=synth.LLAMA, n_layers=6, d_model=16, n_heads=2, n_kv_heads=1, head_dim=8,
                            d_ffn=32, vocab=50, max_pos=64, dtype="f32", max_batch=2, max_seq=16)
    assert cfg.n_kv_heads * cfg.head_dim != cfg.d_model   # D_kv and D told apart
    m = O.OracleModel(cfg, synth.make_weights(cfg, seed=5))
    shapes = synth.weight_shapes(cfg)
    for T, istar in ((1, 2), (3, 4), (5, 6), (2, 1)):
        out = O.skip_kv_fill(m, np.ones((T, cfg.d_model)), np.full(T, istar), np.arange(T))
        flops = bytes_ = 0
        for r, (k, v, sel) in out.items():
            wk, wv = shapes[f"layers.{r - 1}.wk"], shapes[f"layers.{r - 1}.wv"]   # [D_kv, D] each
            flops += len(sel) * 2 * (wk[0] * wk[1] + wv[0] * wv[1])
            bytes_ += (wk[0] * wk[1] + wv[0] * wv[1]) * 2 + len(sel) * (wk[0] + wv[0]) * 2
            assert k.shape == v.shape == (len(sel), cfg.n_kv_heads, cfg.head_dim)
        bytes_ += T * cfg.d_model * 2
        want_f, want_b = bench.fill_micro_work(T, istar, n_layers=cfg.n_layers, d=cfg.d_model,
                                               dkv=cfg.n_kv_heads * cfg.head_dim)
        if istar == cfg.n_layers:   # nothing to fill: no product and no weight read
            assert not out and want_f == 0
            continue
        assert flops == want_f, (T, istar)
        assert bytes_ == want_b, (T, istar)
