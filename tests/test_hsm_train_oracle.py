"""Pins of the HSM training-step oracle (Sec. 4.2, Sec. 5.1 "Training", App. D) against
things other than itself: the independently written inference oracle (Table S1 forward and
the head), central finite differences of the loss, closed forms, and torch.optim.AdamW."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from oracle import hsm_train as HT


def tiny(family, dtype="f32", **kw):
    base = dict(family=family, n_layers=4, d_model=32, n_heads=2, head_dim=16, d_ffn=64, vocab=50, max_pos=32,
                dtype=dtype, norm_eps=1e-5, max_batch=4, max_seq=32, hsm_m1=24, hsm_m2=40)
    base.update(kw)
    return synth.ModelConfig(**base)


def setup(cfg, n=6, seed=0, std=0.2):
    W = synth.make_weights(cfg, seed=seed, std=std, gain_std=0.1 if cfg.dtype == "f32" else None)
    s_i, s_prev, inertia, tgt = synth.hsm_train_batch(cfg, n, seed=seed + 1)
    return W, s_i.double(), s_prev.double(), inertia.double(), tgt.long()


def params_of(W):
    return {k: W[k].double().clone() for k in HT.HSM_PARAMS}


@pytest.mark.parametrize("family,dtype", [(synth.LLAMA, "f32"), (synth.GPT2, "f32"), (synth.LLAMA, "bf16"),
                                          (synth.GPT2, "bf16")])
def test_forward_and_head_match_inference_oracle(family, dtype):
    """Table S1 and the frozen head, written with torch ops here, against the inference
    oracle's numpy restatement (its own conv loop, GEMM-input rounding for bf16)."""
    cfg = tiny(family, dtype)
    W, s_i, s_prev, inertia, _ = setup(cfg)
    om = O.OracleModel(cfg, W)
    bf = dtype == "bf16"
    with torch.no_grad():
        got = HT.hsm_forward(params_of(W), cfg, s_i, s_prev, inertia, bf16=bf).numpy()
        want = om.hsm(s_i.numpy(), s_prev.numpy(), inertia.numpy())
        np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-10)
        lg = HT.head_logits(W, cfg, torch.from_numpy(want), bf16=bf).numpy()
        np.testing.assert_allclose(lg, om.lm_logits(want), rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2])
def test_gradients_match_central_differences(family):
    """Every HSM parameter's gradient against central differences of the fp64 loss."""
    cfg = tiny(family, hsm_eps=1e-6)
    W, s_i, s_prev, inertia, tgt = setup(cfg, n=5)
    p0 = {k: v.numpy() for k, v in params_of(W).items()}
    loss, grads, _, _ = HT.hsm_train_step(W, cfg, s_i, s_prev, inertia, tgt, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1,
                                          params=p0)
    rng = np.random.default_rng(7)

    def L(p):
        with torch.no_grad():
            return float(HT.hsm_loss({k: torch.from_numpy(v) for k, v in p.items()}, W, cfg, s_i, s_prev, inertia,
                                     tgt))

    assert abs(L(p0) - loss) < 1e-13
    h = 1e-6
    for k in HT.HSM_PARAMS:
        flat = p0[k].reshape(-1)
        idx = rng.choice(flat.size, size=min(6, flat.size), replace=False)
        for i in idx:
            pp = {kk: vv.copy() for kk, vv in p0.items()}
            pm = {kk: vv.copy() for kk, vv in p0.items()}
            pp[k].reshape(-1)[i] += h
            pm[k].reshape(-1)[i] -= h
            fd = (L(pp) - L(pm)) / (2 * h)
            g = grads[k].reshape(-1)[i]
            assert abs(fd - g) <= 1e-6 * max(1.0, abs(g)) + 1e-8, (k, int(i), fd, g)
        assert np.abs(grads[k]).max() > 0, k


def test_zero_head_gives_uniform_loss_and_no_gradient():
    """A zero LM head makes every distribution uniform: loss = log V, and nothing flows back."""
    cfg = tiny(synth.LLAMA)
    W, s_i, s_prev, inertia, tgt = setup(cfg)
    W["lm_head"] = torch.zeros_like(W["lm_head"])
    loss, grads, _, _ = HT.hsm_train_step(W, cfg, s_i, s_prev, inertia, tgt, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    assert abs(loss - math.log(cfg.vocab)) < 1e-12
    for k in HT.HSM_PARAMS:
        assert np.abs(grads[k]).max() == 0.0, k


def test_adamw_matches_torch_optim():
    """The written-out AdamW over several steps against torch.optim.AdamW (float64)."""
    rng = np.random.default_rng(3)
    theta = rng.normal(size=(7, 5))
    m = np.zeros_like(theta)
    v = np.zeros_like(theta)
    pt = torch.tensor(theta.copy(), requires_grad=True)
    opt = torch.optim.AdamW([pt], lr=3e-3, betas=(0.8, 0.95), eps=1e-6, weight_decay=0.05)
    for t in range(1, 6):
        g = rng.normal(size=theta.shape) * 10 ** rng.uniform(-4, 0)
        theta, m, v = HT.adamw_update(theta, g, m, v, t, 3e-3, 0.8, 0.95, 1e-6, 0.05)
        pt.grad = torch.tensor(g)
        opt.step()
        np.testing.assert_allclose(theta, pt.detach().numpy(), rtol=1e-13, atol=1e-15)


def test_adamw_first_step_closed_form():
    """t = 1 with zero moments: the bias-corrected ratio is g / (|g| + eps)."""
    g = np.array([3.0, -2e-3, 0.0, 5e-9])
    th = np.array([1.0, 2.0, -1.0, 0.5])
    new, m, v = HT.adamw_update(th, g, np.zeros(4), np.zeros(4), 1, 0.1, 0.9, 0.99, 1e-8, 0.01)
    np.testing.assert_allclose(new, th - 0.1 * 0.01 * th - 0.1 * g / (np.abs(g) + 1e-8), rtol=1e-12)
    np.testing.assert_allclose(m, 0.1 * g)
    np.testing.assert_allclose(v, 0.01 * g * g)


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2])
def test_bf16_mode_stays_within_rounding_of_exact(family):
    """GEMM-input rounding moves the loss and gradients by bf16-sized amounts, not more."""
    cfg = tiny(family, "bf16", d_model=64, head_dim=32, vocab=200, hsm_m1=96, hsm_m2=160)
    W, s_i, s_prev, inertia, tgt = setup(cfg, n=12, std=0.05)
    l64, g64, _, _ = HT.hsm_train_step(W, cfg, s_i, s_prev, inertia, tgt, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    l16, g16, _, _ = HT.hsm_train_step(W, cfg, s_i, s_prev, inertia, tgt, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1, bf16=True)
    assert abs(l16 - l64) <= 1e-2 * abs(l64)
    some_diff = False
    for k in HT.HSM_PARAMS:
        e = np.linalg.norm(g16[k] - g64[k]) / np.linalg.norm(g64[k])
        assert e < 3e-2, (k, e)
        some_diff |= e > 0
    assert some_diff


def test_steps_reduce_the_loss_on_a_fixed_batch():
    """A few AdamW steps on one batch lower its loss (descent property)."""
    cfg = tiny(synth.GPT2)
    W, s_i, s_prev, inertia, tgt = setup(cfg, n=8)
    params, state = None, None
    losses = []
    for t in range(1, 6):
        loss, _, params, state = HT.hsm_train_step(W, cfg, s_i, s_prev, inertia, tgt, 1e-2, 0.9, 0.999, 1e-8, 0.0, t,
                                                   params=params, state=state)
        losses.append(loss)
    assert losses[-1] < losses[0] - 1e-3, losses
