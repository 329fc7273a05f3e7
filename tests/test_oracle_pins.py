"""Pins of the CPU oracle against facts fixed outside it (no GPU).

Each test ties an oracle function to something other than itself: a value the paper
prints, a closed form, a library routine, an invariant of the mathematics, or an
independent evaluation order of the same definitions (tests/torch_reference.py).
"""
import itertools
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import adept_oracle as O
from torch_reference import TorchRef

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_cfg(family, **kw):
    base = dict(family=family, n_layers=4, d_model=32, n_heads=2, head_dim=16, d_ffn=64, vocab=50,
                max_pos=32, n_classes=2 if family == synth.BERT else 0, dtype="f32",
                norm_eps=1e-5, max_batch=4, max_seq=32)
    base.update(kw)
    return synth.ModelConfig(**base)


def model_and_ref(cfg, seed=0, std=0.2, overrides=None):
    W = synth.make_weights(cfg, seed=seed, std=std, gain_std=0.1, overrides=overrides)
    return O.OracleModel(cfg, W), TorchRef(cfg, W), W


# ----------------------------------------------------------------------------- elementary

def test_round_bf16_matches_torch_rne():
    x = synth.normal(3, "bf16-probe", (50000,), std=10.0, dtype=torch.float32)
    # exact ties: 1 + 2^-8 (ties to even -> 1), 1 + 3*2^-8 (-> 1 + 2^-6 ... even)
    ties = torch.tensor([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 2 ** -130, 65504.0], dtype=torch.float32)
    x = torch.cat([x, ties])
    ours = O.round_bf16(x.numpy())
    lib = x.to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(ours, lib)
    assert O.round_bf16(np.array([1 + 2 ** -8]))[0] == 1.0


def test_norms_and_activations_match_library():
    x = synth.normal(1, "x", (7, 24), std=3.0, dtype=torch.float64)
    g = synth.normal(1, "g", (24,), std=0.3, mean=1.0, dtype=torch.float64)
    b = synth.normal(1, "b", (24,), std=0.3, dtype=torch.float64)
    xn, gn, bn = x.numpy(), g.numpy(), b.numpy()
    np.testing.assert_allclose(O.rmsnorm(xn, gn, 1e-5), F.rms_norm(x, (24,), g, 1e-5).numpy(), rtol=1e-12)
    np.testing.assert_allclose(O.layernorm(xn, gn, bn, 1e-5), F.layer_norm(x, (24,), g, b, 1e-5).numpy(),
                               rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(O.gelu_erf(xn), F.gelu(x).numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(O.gelu_tanh(xn), F.gelu(x, approximate="tanh").numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(O.silu(xn), F.silu(x).numpy(), rtol=1e-12, atol=1e-15)


def test_rope_closed_form_and_invariants():
    # d = 2: a single pair rotated by angle pos * theta^0 = pos radians.
    x = np.array([[[1.0, 0.0]]])
    for p in (0, 1, 3):
        y = O.rope(x, np.array([p]), 10000.0)[0, 0]
        np.testing.assert_allclose(y, [math.cos(p), math.sin(p)], atol=1e-15)
    # norm preservation, and <R(q, m), R(k, n)> depends on m - n only.
    q = synth.normal(5, "q", (1, 1, 16), dtype=torch.float64).numpy()
    k = synth.normal(5, "k", (1, 1, 16), dtype=torch.float64).numpy()
    for m_ in (0, 5, 17):
        assert np.isclose(np.linalg.norm(O.rope(q, np.array([m_]), 100.0)), np.linalg.norm(q))
    d1 = np.sum(O.rope(q, np.array([7]), 100.0) * O.rope(k, np.array([3]), 100.0))
    d2 = np.sum(O.rope(q, np.array([24]), 100.0) * O.rope(k, np.array([20]), 100.0))
    assert np.isclose(d1, d2, rtol=1e-12)
    # pairing is (i, i + d/2): feature 0 moves with feature 8, not feature 1.
    e0 = np.zeros((1, 1, 16))
    e0[0, 0, 0] = 1.0
    y = O.rope(e0, np.array([1]), 100.0)[0, 0]
    assert y[8] != 0.0 and y[1] == 0.0


def test_exit_policy_closed_forms():
    """Sec. 4.1: cosine of s_i with the inertia sum of earlier unit states vs delta."""
    e1, e2 = np.eye(4)[0], np.eye(4)[1]
    # earlier states e1 and e2 -> inertia e1+e2; current e1 -> cos 45deg = 1/sqrt2
    inertia = O.unit(np.array([3.0 * e1])) + O.unit(np.array([0.5 * e2]))
    c = O.cosine(np.array([2.0 * e1]), inertia)[0]
    assert np.isclose(c, 1 / math.sqrt(2), rtol=1e-15)
    assert O.cosine(np.array([e1]), np.array([e2]))[0] == 0.0
    assert O.cosine(np.array([np.zeros(4)]), np.array([e1]))[0] == -np.inf
    # scale invariance of the inertia terms: each earlier state counts once
    a = O.unit(np.array([100.0 * e1])) + O.unit(np.array([0.01 * e2]))
    np.testing.assert_allclose(a, [[1.0, 1.0, 0.0, 0.0]])


def test_hsm_conv_matches_torch_conv2d():
    """Table S1: (3, D) -> (1, D), 3x3 kernel, stride 1, padding (0, 1)."""
    X = synth.normal(2, "X", (5, 3, 19), dtype=torch.float64)
    w = synth.normal(2, "w", (3, 3), dtype=torch.float64)
    b = torch.tensor([0.25], dtype=torch.float64)
    ref = F.conv2d(X[:, None], w[None, None], b, stride=1, padding=(0, 1))[:, 0, 0]
    np.testing.assert_allclose(O.hsm_conv(X.numpy(), w.numpy(), 0.25), ref.numpy(), rtol=1e-13, atol=1e-14)


def test_hsm_param_counts_match_paper():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "hsm_param_counts.txt")) if l.strip() and not l.startswith("#")]
    assert len(rows) == 4
    for name, d, m1, m2, copies, printed in rows:
        n = int(copies) * O.hsm_param_count(int(d), int(m1), int(m2))
        assert round(n / 1e6) == int(printed), name
    # Table S1 widths give 72 D^2 weights
    assert O.hsm_param_count(10, 40, 80) == 72 * 100


def test_hsm_zero_mlp_closed_form():
    """FC weights zero, eps 0: s~ = RMSNorm_g2(b4) + c0, c0 = the 1-D correlation of the
    (identical) normalised rows with the column-summed kernel, plus the conv bias."""
    cfg = small_cfg(synth.LLAMA, hsm_eps=0.0)
    W = synth.make_weights(cfg, seed=4, std=0.2, gain_std=0.1)
    for n in ("hsm.fc1_w", "hsm.fc2_w", "hsm.fc3_w", "hsm.fc4_w"):
        W[n] = torch.zeros_like(W[n])
    m = O.OracleModel(cfg, W)
    x = synth.normal(4, "s", (1, 32), dtype=torch.float64).numpy()
    out = m.hsm(x, 3.0 * x, 0.5 * x)[0]
    g0, g2 = m.w["hsm.g0"], m.w["hsm.g2"]
    xn = x[0] / math.sqrt(np.mean(x[0] ** 2)) * g0
    k = m.w["hsm.conv_w"].sum(axis=0)
    c0 = np.correlate(np.pad(xn, 1), k, mode="valid") + m.w["hsm.conv_b"][0]
    b4 = m.w["hsm.fc4_b"]
    expect = b4 / math.sqrt(np.mean(b4 ** 2)) * g2 + c0
    np.testing.assert_allclose(out, expect, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- whole pass

@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2, synth.BERT])
def test_full_depth_matches_standard_transformer(family):
    """delta = +inf (and forced exit N) reduces ADEPT to the plain full-depth model."""
    cfg = small_cfg(family)
    m, ref, _ = model_and_ref(cfg, seed=11)
    tokens = synth.make_tokens(11, 3, 9, cfg.vocab).numpy()
    want = ref.full_forward(torch.as_tensor(tokens)).numpy()
    for forced in (None, np.full(27, cfg.n_layers)):
        cache = O.OracleCache(cfg, 3, 16)
        r = O.prefill(m, cache, tokens, float("inf"), forced)
        assert np.all(r.exit_layer == cfg.n_layers)
        assert np.all(np.isnan(r.sim[:, 0])) and np.all(np.isnan(r.sim[:, -1]))
        np.testing.assert_allclose(r.final.reshape(want.shape), want, rtol=1e-10, atol=1e-10)
        head_in = want[:, 0] if family == synth.BERT else want[:, -1]
        np.testing.assert_allclose(r.logits, ref.head(torch.as_tensor(head_in)).numpy(), rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2])
def test_full_depth_decode_matches_recompute(family):
    """Cached decode steps == a no-cache full recompute of the longer sequence."""
    cfg = small_cfg(family)
    m, ref, _ = model_and_ref(cfg, seed=12)
    tokens = synth.make_tokens(12, 2, 10, cfg.vocab).numpy()
    cache = O.OracleCache(cfg, 2, 16)
    O.prefill(m, cache, tokens[:, :6], float("inf"))
    for t in range(6, 10):
        r = O.decode_step(m, cache, tokens[:, t], float("inf"))
        want = ref.full_forward(torch.as_tensor(tokens[:, :t + 1])).numpy()[:, -1]
        np.testing.assert_allclose(r.final, want, rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(r.logits, ref.head(torch.as_tensor(want)).numpy(), rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("hsm_mode", ["hsm", "identity"])
def test_brute_force_token_major_unfold(hsm_mode):
    """Every forced-exit assignment in {2, 3}^5 on N=3, D=8, 2 heads, 5 tokens: the layer-major
    parallel pass (App. I) equals a one-token-at-a-time unfold built from library ops,
    in final states, exit layers and every cached K/V entry of every layer."""
    cfg = small_cfg(synth.LLAMA, n_layers=3, d_model=8, n_heads=2, head_dim=4, d_ffn=16, vocab=11)
    m, ref, _ = model_and_ref(cfg, seed=13, std=0.4)
    tokens = synth.make_tokens(13, 1, 5, cfg.vocab).numpy()
    for assign in itertools.product([2, 3], repeat=5):
        forced = np.array(assign)
        cache = O.OracleCache(cfg, 1, 8)
        r = O.prefill(m, cache, tokens, 0.5, forced, hsm_mode=hsm_mode)
        fin, el, K, V = ref.token_major(tokens[0], forced, hsm_mode)
        np.testing.assert_array_equal(r.exit_layer, el.numpy())
        np.testing.assert_allclose(r.final, fin.numpy(), rtol=1e-11, atol=1e-12)
        for i in range(1, 4):
            for j in range(5):
                np.testing.assert_allclose(cache.K[i - 1][0, j], K[i][j].numpy(), rtol=1e-11, atol=1e-12)
                np.testing.assert_allclose(cache.V[i - 1][0, j], V[i][j].numpy(), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2, synth.BERT])
def test_forced_exit_fills_projection_of_mapped_state(family):
    """Forced exit at l: for every r > l the cache holds layer r's K/V projection of s~_N
    (norm, W_K / W_V, bias, RoPE at the token's position, evaluated with library ops)."""
    cfg = small_cfg(family, n_layers=5)
    m, ref, _ = model_and_ref(cfg, seed=14)
    tokens = synth.make_tokens(14, 2, 6, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(14, 12, 2, 5).numpy()
    cache = O.OracleCache(cfg, 2, 8)
    r = O.prefill(m, cache, tokens, 0.0, forced)
    np.testing.assert_array_equal(r.exit_layer, forced)
    pos = np.tile(np.arange(6), 2)
    seq = np.repeat(np.arange(2), 6)
    checked = 0
    for t in range(12):
        for rr in range(forced[t] + 1, 6):
            k, v = ref.kv(rr, torch.as_tensor(r.final[t]), torch.tensor(pos[t]))
            np.testing.assert_allclose(cache.K[rr - 1][seq[t], pos[t]], k.numpy(), rtol=1e-11, atol=1e-12)
            np.testing.assert_allclose(cache.V[rr - 1][seq[t], pos[t]], v.numpy(), rtol=1e-11, atol=1e-12)
            checked += 1
    assert checked > 0


def test_degenerate_identity_layers_exit_at_first_eligible_layer():
    """W_O = W_down = 0 makes every layer the identity: s_i = s_0, the cosine with the
    inertia is exactly 1 and every token leaves at layer 2 for any delta <= 1."""
    cfg = small_cfg(synth.LLAMA, n_layers=5)
    W = synth.make_weights(cfg, seed=15, std=0.2, gain_std=0.1)
    for l in range(cfg.n_layers):
        W[f"layers.{l}.wo"] = torch.zeros_like(W[f"layers.{l}.wo"])
        W[f"layers.{l}.w_down"] = torch.zeros_like(W[f"layers.{l}.w_down"])
    m = O.OracleModel(cfg, W)
    tokens = synth.make_tokens(15, 2, 7, cfg.vocab).numpy()
    cache = O.OracleCache(cfg, 2, 8)
    r = O.prefill(m, cache, tokens, 1.0 - 1e-12)
    assert np.all(r.exit_layer == 2)
    np.testing.assert_allclose(r.sim[:, 1], 1.0, atol=1e-14)
    s0 = m.embed(tokens.reshape(-1), np.tile(np.arange(7), 2))
    unit0 = O.unit(s0)
    np.testing.assert_allclose(r.final, m.hsm(s0, s0, unit0), rtol=1e-12, atol=1e-12)
    # delta above 1 never exits
    r2 = O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, 1.0 + 1e-9)
    assert np.all(r2.exit_layer == cfg.n_layers)


def test_threshold_minus_two_exits_at_layer_two_and_inf_never():
    cfg = small_cfg(synth.GPT2)
    m, _, _ = model_and_ref(cfg, seed=16)
    tokens = synth.make_tokens(16, 2, 5, cfg.vocab).numpy()
    assert np.all(O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, -2.0).exit_layer == 2)
    assert np.all(O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, np.inf).exit_layer == cfg.n_layers)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2])
def test_prefill_then_decode_equals_longer_prefill(family):
    cfg = small_cfg(family, n_layers=5)
    m, _, _ = model_and_ref(cfg, seed=17)
    tokens = synth.make_tokens(17, 2, 8, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(17, 16, 2, 5).numpy().reshape(2, 8)
    c1 = O.OracleCache(cfg, 2, 16)
    long = O.prefill(m, c1, tokens, 0.0, forced)
    c2 = O.OracleCache(cfg, 2, 16)
    O.prefill(m, c2, tokens[:, :7], 0.0, forced[:, :7])
    step = O.decode_step(m, c2, tokens[:, 7], 0.0, forced[:, 7])
    np.testing.assert_allclose(step.logits, long.logits, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(step.final, long.final.reshape(2, 8, -1)[:, 7], rtol=1e-10, atol=1e-12)
    for l in range(cfg.n_layers):
        np.testing.assert_allclose(c2.K[l][:, :8], c1.K[l][:, :8], rtol=1e-10, atol=1e-12)


def test_batch_independence():
    cfg = small_cfg(synth.LLAMA, n_layers=5)
    m, _, _ = model_and_ref(cfg, seed=18)
    tokens = synth.make_tokens(18, 3, 6, cfg.vocab).numpy()
    both = O.prefill(m, O.OracleCache(cfg, 3, 8), tokens, 0.3)
    for b in range(3):
        one = O.prefill(m, O.OracleCache(cfg, 1, 8), tokens[b:b + 1], 0.3)
        np.testing.assert_array_equal(one.exit_layer, both.exit_layer.reshape(3, 6)[b])
        np.testing.assert_allclose(one.final, both.final.reshape(3, 6, -1)[b], rtol=1e-12, atol=1e-13)


def test_forced_exit_validation():
    cfg = small_cfg(synth.LLAMA)
    m, _, _ = model_and_ref(cfg)
    tokens = synth.make_tokens(0, 1, 3, cfg.vocab).numpy()
    with pytest.raises(ValueError):
        O.prefill(m, O.OracleCache(cfg, 1, 8), tokens, 0.5, np.array([1, 0, 0]))
    with pytest.raises(ValueError):
        O.prefill(m, O.OracleCache(cfg, 1, 8), tokens, 0.5, np.array([0, 5, 0]))


def test_bf16_contract_rounds_cached_kv():
    cfg = small_cfg(synth.LLAMA, dtype="bf16")
    W = synth.make_weights(cfg, seed=19, std=0.2)
    m = O.OracleModel(cfg, W)
    for t in W.values():
        assert t.dtype == torch.bfloat16
    cache = O.OracleCache(cfg, 1, 8)
    O.prefill(m, cache, synth.make_tokens(19, 1, 5, cfg.vocab).numpy(), 0.2)
    k = cache.K[2][0, :5]
    np.testing.assert_array_equal(k, O.round_bf16(k))


def test_synth_generator_is_deterministic_and_normal():
    a = synth.normal(0, "w", (200000,), std=0.02, dtype=torch.float64)
    b = synth.normal(0, "w", (200000,), std=0.02, dtype=torch.float64)
    assert torch.equal(a, b)
    assert abs(a.mean().item()) < 3 * 0.02 / math.sqrt(2e5) * 2
    assert abs(a.std().item() / 0.02 - 1) < 0.01
    c = synth.normal(0, "w2", (10,), dtype=torch.float64)
    assert not torch.equal(a[:10] / 0.02, c)
    # chunk boundary does not change values
    x = synth.normal(7, "big", (synth._CHUNK + 5,), dtype=torch.float64)
    y = synth.normal(7, "big", (synth._CHUNK + 5,), dtype=torch.float64)
    assert torch.equal(x[-10:], y[-10:])
    t = synth.forced_exits_truncnorm(0, 20000, 24.0, 4.0, 8, 32)
    assert t.min() >= 8 and t.max() <= 32 and abs(t.double().mean().item() - 23.79) < 0.15
    u = synth.forced_exits_uniform(0, 20000, 4, 12)
    assert u.min() == 4 and u.max() == 12


def test_synth_training_batches_follow_their_recipe():
    """HSM training examples: s_i - s_{i-1} ~ N(0, (0.3 std)^2); I = (k - 1) unit(s_{i-1}) + noise
    with k in [2, N - 1]; targets in [0, V); encoder examples add s_N - s_i ~ N(0, (0.5 std)^2) and
    labels in [0, n_classes) for the first n_cls rows."""
    cfg = synth.bert_base_config(n_layers=12)
    s_i, s_prev, inertia, tgt = synth.hsm_train_batch(cfg, 4000, seed=3, std=0.5)
    assert abs(s_prev.std().item() / 0.5 - 1) < 0.01
    assert abs((s_i - s_prev).std().item() / 0.15 - 1) < 0.01
    u = s_prev / s_prev.norm(dim=1, keepdim=True)
    k1 = (inertia * u).sum(1)   # (k - 1) + the noise's projection
    assert k1.min().item() > 1 - 0.6 and k1.max().item() < cfg.n_layers - 2 + 0.6
    assert int(tgt.min()) >= 0 and int(tgt.max()) < cfg.vocab
    a, b, c, s_fin, lab = synth.hsm_cls_batch(cfg, 4000, 64, seed=3, std=0.5)
    assert torch.equal(a, s_i) and torch.equal(b, s_prev) and torch.equal(c, inertia)
    assert abs((s_fin - s_i).std().item() / 0.25 - 1) < 0.01
    assert lab.shape == (64,) and lab.dtype == torch.int32
    assert int(lab.min()) == 0 and int(lab.max()) == cfg.n_classes - 1


# ----------------------------------------------------------------------------- threshold calibration

def test_rdc_closed_forms():
    """RDC = 1 - sum(depth) / (T N) (Sec. 5.1): every token at layer 2 -> 1 - 2/N, full
    depth -> 0; a hand example."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, _, _ = model_and_ref(cfg, seed=41)
    tokens = synth.make_tokens(41, 2, 7, cfg.vocab).numpy()
    lo = O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, -2.0)
    hi = O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, np.inf)
    assert O.reduction_in_computation(lo.exit_layer, 6) == pytest.approx(1 - 2 / 6, abs=1e-15)
    assert O.reduction_in_computation(hi.exit_layer, 6) == 0.0
    assert O.reduction_in_computation(np.array([2, 6, 4, 4]), 8) == pytest.approx(1 - 16 / 32, abs=1e-15)


def test_calibration_bisection_against_brute_force():
    """Bisection on delta lands on a threshold whose prompt-pass RDC equals an attainable
    target; the brute-force scan over a delta grid shows the RDC falling with delta (a
    stricter threshold keeps tokens longer) and gives that target."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, _, _ = model_and_ref(cfg, seed=42, std=0.05)
    tokens = synth.make_tokens(42, 2, 12, cfg.vocab).numpy()
    grid = np.linspace(-1.0, 1.0, 41)
    rdc = np.array([O.reduction_in_computation(O.prefill(m, O.OracleCache(cfg, 2, 16), tokens, d).exit_layer, 6)
                    for d in grid])
    assert np.all(np.diff(rdc) <= 1e-12)                      # non-increasing in delta
    assert rdc[0] == pytest.approx(1 - 2 / 6) and rdc[-1] < rdc[0]
    mids = [r for r in np.unique(rdc) if 0.0 < r < 1 - 2 / 6]
    assert mids, "the scan should reach intermediate reductions"
    target = mids[len(mids) // 2]
    d, r, hist = O.calibrate_threshold(m, tokens, target, tol=1e-12, max_iter=30)
    assert r == pytest.approx(target, abs=1e-12)
    # the returned threshold reproduces the reduction in a fresh pass
    again = O.reduction_in_computation(O.prefill(m, O.OracleCache(cfg, 2, 16), tokens, d).exit_layer, 6)
    assert again == pytest.approx(target, abs=1e-12)
    # bisection: each pass halves the bracket, which always holds the result
    lo, hi = -1.0, 1.0
    for dd, rr in hist[:-1]:
        assert dd == pytest.approx(0.5 * (lo + hi), abs=0)
        if rr > target:
            lo = dd
        else:
            hi = dd
    assert lo <= d <= hi


def test_calibration_unreachable_target_ends_at_the_bound():
    """A target above the largest attainable reduction (1 - 2/N) drives delta to the lower
    end of the bracket, with every token leaving at layer 2."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, _, _ = model_and_ref(cfg, seed=43)
    tokens = synth.make_tokens(43, 1, 6, cfg.vocab).numpy()
    d, r, hist = O.calibrate_threshold(m, tokens, 0.99, lo=-1.0, hi=1.0, max_iter=12)
    assert len(hist) == 12
    assert d == pytest.approx(-1.0 + 2.0 ** -11, abs=1e-15)   # passes at 0, -1/2, ..., -1 + 2^-11
    assert r == pytest.approx(1 - 2 / 6)


# ----------------------------------------------------------------------------- exit-rule variants

def _layer_states(ref, tokens):
    """Full-depth states s_0..s_N of every token from the independent torch model
    ([N + 1, B, P, D], float64)."""
    c = ref.c
    tokens = torch.as_tensor(tokens)
    B, P = tokens.shape
    pos = torch.arange(P).expand(B, P)
    h = ref.embed(tokens, pos)
    out = [h]
    for i in range(1, c.n_layers + 1):
        q = ref.q(i, h, pos).transpose(1, 2)
        k, v = ref.kv(i, h, pos)
        rep = c.n_heads // c.n_kv_heads
        k = k.repeat_interleave(rep, dim=2).transpose(1, 2)
        v = v.repeat_interleave(rep, dim=2).transpose(1, 2)
        a = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        h = ref.after_attn(i, h, a.transpose(1, 2).flatten(-2))
        out.append(h)
    return torch.stack(out).numpy()


def _cos(a, b):
    return np.sum(a * b, -1) / (np.linalg.norm(a, axis=-1) * np.linalg.norm(b, axis=-1))


@pytest.mark.parametrize("metric", ["global", "local", "both"])
def test_recorded_similarities_match_full_depth_states(metric):
    """At delta = +inf nothing leaves, so the recorded similarity at layer i (2 <= i <= N-1)
    is the metric on the plain full-depth states: global cos(s_i, sum_{d<i} s_hat_d) (Eq. 7),
    local cos(s_i, s_{i-1}), both their minimum."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, ref, _ = model_and_ref(cfg, seed=51)
    tokens = synth.make_tokens(51, 2, 7, cfg.vocab).numpy()
    S = _layer_states(ref, tokens)          # [N+1, B, P, D]
    r = O.prefill(m, O.OracleCache(cfg, 2, 8), tokens, np.inf, metric=metric)
    for i in range(2, cfg.n_layers):
        inertia = sum(S[d] / np.linalg.norm(S[d], axis=-1, keepdims=True) for d in range(1, i))
        g = _cos(S[i], inertia).reshape(-1)
        l = _cos(S[i], S[i - 1]).reshape(-1)
        want = g if metric == "global" else l if metric == "local" else np.minimum(g, l)
        np.testing.assert_allclose(r.sim[:, i - 1], want, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("metric", ["global", "local", "both"])
def test_single_token_sequences_exit_at_the_first_crossing(metric):
    """A one-token sequence is computed normally until it leaves, so its exit layer is the
    first i in [2, N-1] where its full-depth metric reaches delta (N if none)."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, ref, _ = model_and_ref(cfg, seed=52, std=0.05)
    tokens = synth.make_tokens(52, 4, 1, cfg.vocab).numpy()
    S = _layer_states(ref, tokens)[:, :, 0]    # [N+1, B, D]
    probe = np.unique(O.prefill(m, O.OracleCache(cfg, 4, 2), tokens, np.inf, metric=metric).sim[:, 1:cfg.n_layers - 1])
    # thresholds half-way between neighbouring similarities: no decision sits on a tie
    for k in (len(probe) // 4, len(probe) // 2, 3 * len(probe) // 4):
        delta = 0.5 * (probe[k - 1] + probe[k])
        r = O.prefill(m, O.OracleCache(cfg, 4, 2), tokens, float(delta), metric=metric)
        for b in range(4):
            want = cfg.n_layers
            for i in range(2, cfg.n_layers):
                inertia = sum(S[d, b] / np.linalg.norm(S[d, b]) for d in range(1, i))
                g, l = _cos(S[i, b], inertia), _cos(S[i, b], S[i - 1, b])
                v = g if metric == "global" else l if metric == "local" else min(g, l)
                if v >= delta:
                    want = i
                    break
            assert r.exit_layer[b] == want


def test_all_at_once_sequences_leave_with_their_last_token():
    """All-at-once (App. H.2): every token of a sequence leaves at the layer where the
    sequence's last prompt token first reaches delta on the full-depth states (the
    sequence is complete until then), N if it never does."""
    cfg = small_cfg(synth.GPT2, n_layers=6)
    m, ref, _ = model_and_ref(cfg, seed=53, std=0.05)
    B, P = 3, 6
    tokens = synth.make_tokens(53, B, P, cfg.vocab).numpy()
    S = _layer_states(ref, tokens)[:, :, P - 1]   # last token, [N+1, B, D]
    probe = np.unique(O.prefill(m, O.OracleCache(cfg, B, P), tokens, np.inf).sim.reshape(B, P, -1)[:, P - 1,
                                                                                                   1:cfg.n_layers - 1])
    for k in (len(probe) // 4, 3 * len(probe) // 5):
        delta = 0.5 * (probe[k - 1] + probe[k])
        r = O.prefill(m, O.OracleCache(cfg, B, P), tokens, float(delta), all_at_once=True)
        ex = r.exit_layer.reshape(B, P)
        for b in range(B):
            want = cfg.n_layers
            for i in range(2, cfg.n_layers):
                inertia = sum(S[d, b] / np.linalg.norm(S[d, b]) for d in range(1, i))
                if _cos(S[i, b], inertia) >= delta:
                    want = i
                    break
            assert np.all(ex[b] == want)


def test_encoder_stop_entirely_matches_independent_masked_model():
    """Encoder "stop entirely" (Sec. 4.3, downstream tasks) with forced exits against a
    token-subset forward of the independent torch model: at each layer only the tokens
    still active are computed, and attend to each other only (bidirectional); an exiting
    token's output is the HSM of (s_i, s_{i-1}, inertia before s_hat_i)."""
    cfg = small_cfg(synth.BERT, n_layers=5)
    m, ref, _ = model_and_ref(cfg, seed=54)
    P = 7
    tokens = synth.make_tokens(54, 1, P, cfg.vocab).numpy()
    forced = np.array([2, 5, 3, 4, 2, 5, 3])
    r = O.prefill(m, O.OracleCache(cfg, 1, 8), tokens, 0.5, forced, stop_entirely=True)
    np.testing.assert_array_equal(r.exit_layer, forced)
    # the torch side
    tk = torch.as_tensor(tokens)
    pos = torch.arange(P)[None]
    h = ref.embed(tk, pos)[0]
    inertia = torch.zeros_like(h)
    final = torch.zeros_like(h)
    active = np.ones(P, dtype=bool)
    for i in range(1, cfg.n_layers + 1):
        A = np.nonzero(active)[0]
        hA = h[A][None]
        q = ref.q(i, hA, pos[:, A]).transpose(1, 2)
        k, v = ref.kv(i, hA, pos[:, A])
        a = F.scaled_dot_product_attention(q, k.transpose(1, 2), v.transpose(1, 2))
        s_new = ref.after_attn(i, hA, a.transpose(1, 2).flatten(-2))[0]
        ex = (forced[A] == i) if 2 <= i <= cfg.n_layers - 1 else np.zeros(len(A), dtype=bool)
        I_before = inertia[A].clone()
        inertia[A] = I_before + s_new / s_new.norm(dim=-1, keepdim=True)
        for kk in np.nonzero(ex)[0]:
            j = A[kk]
            final[j] = ref.hsm(s_new[kk], h[j], I_before[kk])
        h[A] = s_new
        active[A[ex]] = False
    final[active] = h[active]
    np.testing.assert_allclose(r.final, final.numpy(), rtol=1e-10, atol=1e-10)
    # the classifier reads position 0's state
    np.testing.assert_allclose(r.logits[0], ref.head(final[0][None]).numpy()[0], rtol=1e-10, atol=1e-10)


# ----------------------------------------------------------------------------- skipped-layer fill rows

def test_skip_kv_fill_rows_are_exactly_the_skipped_layers():
    """O.skip_kv_fill (Sec. 4.3 KV generation): token j is filled at exactly the layers
    r = i*_j + 1 .. N (never at its exit layer i*_j itself, nothing for i*_j = N), and each
    entry equals layer r's K/V projection of s~ evaluated with library ops (TorchRef.kv)."""
    for family in (synth.LLAMA, synth.GPT2, synth.BERT):
        cfg = small_cfg(family, n_layers=5)
        m, ref, _ = model_and_ref(cfg, seed=22)
        n = 12
        mapped = synth.normal(22, "mapped", (n, cfg.d_model), std=1.0, dtype=torch.float64).numpy()
        exit_layer = np.array([1, 2, 3, 4, 5, 5, 2, 3, 1, 4, 5, 2])
        pos = np.array([0, 3, 1, 7, 2, 5, 4, 6, 9, 8, 11, 10])
        out = O.skip_kv_fill(m, mapped, exit_layer, pos)
        filled = {j: set() for j in range(n)}
        for r, (k, v, sel) in out.items():
            assert 2 <= r <= cfg.n_layers
            for a, j in enumerate(sel):
                filled[int(j)].add(r)
                kw, vw = ref.kv(r, torch.as_tensor(mapped[j]), torch.tensor(int(pos[j])))
                np.testing.assert_allclose(k[a], kw.numpy(), rtol=1e-11, atol=1e-12)
                np.testing.assert_allclose(v[a], vw.numpy(), rtol=1e-11, atol=1e-12)
        for j in range(n):
            assert filled[j] == set(range(int(exit_layer[j]) + 1, cfg.n_layers + 1)), (family, j)


# ----------------------------------------------------------------------------- bf16 contract

def _bf16_pair(family):
    cfg = small_cfg(family, n_layers=4, dtype="bf16")
    W = synth.make_weights(cfg, seed=21, std=0.2, gain_std=0.1)
    return cfg, O.OracleModel(cfg, W), TorchRef(cfg, W, bf16=True)


def _bf16_gap(cfg, m, ref, tokens, forced):
    """Largest relative gap between the oracle's bf16 pass and the reference's bf16 statement
    of the contract, over final states, logits and every cached K/V entry."""
    gaps = []
    rel = lambda a, b: float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))  # noqa: E731
    if cfg.family == synth.BERT:
        cache = O.OracleCache(cfg, 1, 8)
        r = O.prefill(m, cache, tokens, np.inf)
        want = ref.full_forward(torch.as_tensor(tokens))[0]
        gaps.append(rel(r.final, want.numpy()))
        gaps.append(rel(r.logits, ref.head(want[0:1]).numpy()))
        pos = torch.arange(tokens.shape[1])
        h = ref.embed(torch.as_tensor(tokens[0]), pos)
        for i in range(1, cfg.n_layers + 1):     # layer inputs again, for the cached K/V
            k, v = ref.kv(i, h, pos)
            gaps.append(rel(cache.K[i - 1][0, :tokens.shape[1]], k.numpy()))
            gaps.append(rel(cache.V[i - 1][0, :tokens.shape[1]], v.numpy()))
            q = ref.q(i, h, pos).transpose(0, 1)
            a = F.scaled_dot_product_attention(q, k.transpose(0, 1), v.transpose(0, 1))
            h = ref.after_attn(i, h, a.transpose(0, 1).flatten(-2))
        return max(gaps)
    cache = O.OracleCache(cfg, 1, 8)
    r = O.prefill(m, cache, tokens, 0.5, forced)
    fin, el, K, V = ref.token_major(tokens[0], forced)
    np.testing.assert_array_equal(r.exit_layer, el.numpy())
    gaps.append(rel(r.final, fin.numpy()))
    gaps.append(rel(r.logits, ref.head(fin[-1:]).numpy()))
    for i in range(1, cfg.n_layers + 1):
        for j in range(tokens.shape[1]):
            gaps.append(rel(cache.K[i - 1][0, j], K[i][j].numpy()))
            gaps.append(rel(cache.V[i - 1][0, j], V[i][j].numpy()))
    return max(gaps)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2, synth.BERT])
def test_bf16_contract_matches_independent_statement(family):
    """bf16 models: the oracle's pass (decoders: forced exits through the mapper and the fills;
    the encoder: full depth) equals the torch reference with the contract's rounding points
    applied by torch's own bf16 cast, to ~1e-12, in final states, logits and every cached K/V
    entry."""
    cfg, m, ref = _bf16_pair(family)
    tokens = synth.make_tokens(21, 1, 6, cfg.vocab).numpy()
    forced = np.array([2, 4, 3, 2, 4, 3])
    assert _bf16_gap(cfg, m, ref, tokens, forced) < 1e-12


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2, synth.BERT])
def test_bf16_contract_pin_fails_on_a_missing_or_extra_rounding_point(family, monkeypatch):
    """The agreement above has teeth: dropping any single rounding point the oracle takes
    during the pass (each call of OracleModel.rb in turn), or adding one on the residual
    stream, moves the oracle away from the reference by far more than 1e-12."""
    cfg, m, ref = _bf16_pair(family)
    tokens = synth.make_tokens(21, 1, 6, cfg.vocab).numpy()
    forced = np.array([2, 4, 3, 2, 4, 3])
    rb = O.OracleModel.rb
    calls = {"n": 0, "skip": -1}

    def counting_rb(self, x):
        calls["n"] += 1
        return x if calls["n"] - 1 == calls["skip"] else rb(self, x)

    monkeypatch.setattr(O.OracleModel, "rb", counting_rb)
    _bf16_gap(cfg, m, ref, tokens, forced)
    total = calls["n"]
    assert total >= 8 * cfg.n_layers
    for k in range(total):
        calls["n"], calls["skip"] = 0, k
        assert _bf16_gap(cfg, m, ref, tokens, forced) > 1e-6, f"rounding point {k} of {total} has no effect"
    monkeypatch.setattr(O.OracleModel, "rb", rb)
    body = O.layer_body
    monkeypatch.setattr(O, "layer_body", lambda mm, *a, **kw: O.round_bf16(body(mm, *a, **kw)))
    assert _bf16_gap(cfg, m, ref, tokens, forced) > 1e-6
