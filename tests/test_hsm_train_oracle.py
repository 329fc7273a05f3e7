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


# ---------------------------------------------------------------------------
# encoders: similarity loss + task loss (Sec. 4.3)
# ---------------------------------------------------------------------------

def tiny_bert(dtype="f32", **kw):
    base = dict(max_pos=32, n_classes=3, norm_eps=1e-12)
    base.update(kw)
    return tiny(synth.BERT, dtype, **base)


def setup_cls(cfg, n=6, n_cls=3, seed=0, std=0.2):
    W = synth.make_weights(cfg, seed=seed, std=std, gain_std=0.1 if cfg.dtype == "f32" else None)
    s_i, s_prev, inertia, s_fin, lab = synth.hsm_cls_batch(cfg, n, n_cls, seed=seed + 1)
    return W, s_i.double(), s_prev.double(), inertia.double(), s_fin.double(), lab.long()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_cls_head_matches_inference_oracle(dtype):
    """The pooler + classifier written with torch ops against the inference oracle's numpy
    restatement of the encoder's classification head."""
    cfg = tiny_bert(dtype)
    W, s_i, s_prev, inertia, _, _ = setup_cls(cfg)
    om = O.OracleModel(cfg, W)
    st = om.hsm(s_i.numpy(), s_prev.numpy(), inertia.numpy())
    with torch.no_grad():
        got = HT.cls_head_logits(W, cfg, torch.from_numpy(st), bf16=dtype == "bf16").numpy()
    np.testing.assert_allclose(got, om.cls_logits(st), rtol=1e-10, atol=1e-10)


def test_similarity_loss_is_mean_cosine_distance():
    """With no labelled rows the loss is the mean cosine distance (scipy) between the
    inference oracle's mapped states and the final states."""
    from scipy.spatial.distance import cosine
    cfg = tiny_bert()
    W, s_i, s_prev, inertia, s_fin, _ = setup_cls(cfg, n=7)
    om = O.OracleModel(cfg, W)
    st = om.hsm(s_i.numpy(), s_prev.numpy(), inertia.numpy())
    want = np.mean([cosine(st[i], s_fin[i].numpy()) for i in range(7)])
    with torch.no_grad():
        got = float(HT.hsm_cls_loss(params_of(W), W, cfg, s_i, s_prev, inertia, s_fin, []))
    assert abs(got - want) < 1e-12


@pytest.mark.parametrize("sign", [1.0, -1.0])
def test_aligned_targets_are_stationary(sign):
    """Targets along (+) or against (-) the mapped states: loss 0 or 2, and the gradient of
    1 - cos vanishes at both extremes."""
    cfg = tiny_bert()
    W, s_i, s_prev, inertia, _, _ = setup_cls(cfg, n=5)
    om = O.OracleModel(cfg, W)
    st = om.hsm(s_i.numpy(), s_prev.numpy(), inertia.numpy())
    scale = sign * (0.5 + np.arange(5))[:, None]
    loss, grads, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, torch.from_numpy(st * scale), [], 1.0,
                                              1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    assert abs(loss - (1.0 - sign)) < 1e-12
    for k in HT.HSM_PARAMS:
        assert np.abs(grads[k]).max() < 1e-9, k


def test_zero_target_row_adds_one_and_no_gradient():
    """A zero final state has no direction: its cosine is taken as 0 (term 1), with no gradient."""
    cfg = tiny_bert()
    W, s_i, s_prev, inertia, s_fin, _ = setup_cls(cfg, n=4)
    z = s_fin.clone()
    z[2] = 0.0
    l_all, g_all, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, z, [], 1.0, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    keep = [0, 1, 3]
    l3, g3, _, _ = HT.hsm_cls_train_step(W, cfg, s_i[keep], s_prev[keep], inertia[keep], z[keep], [], 1.0, 1e-3, 0.9,
                                         0.999, 1e-8, 0.0, 1)
    assert abs(l_all - (3 * l3 + 1.0) / 4) < 1e-12
    for k in HT.HSM_PARAMS:
        np.testing.assert_allclose(g_all[k], 0.75 * g3[k], rtol=1e-9, atol=1e-15)


def test_two_class_task_loss_is_binary_cross_entropy():
    """Two classes: the task term is torch's binary cross-entropy with logits on z1 - z0 of the
    inference oracle's classifier logits, times cls_weight."""
    cfg = tiny_bert(n_classes=2)
    W, s_i, s_prev, inertia, s_fin, lab = setup_cls(cfg, n=6, n_cls=4)
    om = O.OracleModel(cfg, W)
    st = om.hsm(s_i.numpy(), s_prev.numpy(), inertia.numpy())
    z = torch.from_numpy(om.cls_logits(st[:4]))
    bce = F_bce(z[:, 1] - z[:, 0], lab.double())
    p = params_of(W)
    with torch.no_grad():
        l0 = float(HT.hsm_cls_loss(p, W, cfg, s_i, s_prev, inertia, s_fin, lab, cls_weight=0.0))
        l1 = float(HT.hsm_cls_loss(p, W, cfg, s_i, s_prev, inertia, s_fin, lab, cls_weight=0.6))
    assert abs((l1 - l0) - 0.6 * bce) < 1e-12


def F_bce(x, y):
    return float(torch.nn.functional.binary_cross_entropy_with_logits(x, y))


@pytest.mark.parametrize("n_cls", [0, 3, 5])
def test_cls_gradients_match_central_differences(n_cls):
    """Every HSM parameter's gradient of similarity + weighted task loss against central
    differences (no labelled rows, some, all)."""
    cfg = tiny_bert(hsm_eps=1e-6)
    W, s_i, s_prev, inertia, s_fin, lab = setup_cls(cfg, n=5, n_cls=n_cls)
    p0 = {k: v.numpy() for k, v in params_of(W).items()}
    loss, grads, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, s_fin, lab, 0.7, 1e-3, 0.9, 0.999, 1e-8,
                                              0.0, 1, params=p0)
    rng = np.random.default_rng(11)

    def L(p):
        with torch.no_grad():
            return float(HT.hsm_cls_loss({k: torch.from_numpy(v) for k, v in p.items()}, W, cfg, s_i, s_prev, inertia,
                                         s_fin, lab, 0.7))

    assert abs(L(p0) - loss) < 1e-13
    h = 1e-6
    for k in HT.HSM_PARAMS:
        flat = p0[k].reshape(-1)
        for i in rng.choice(flat.size, size=min(5, flat.size), replace=False):
            pp = {kk: vv.copy() for kk, vv in p0.items()}
            pm = {kk: vv.copy() for kk, vv in p0.items()}
            pp[k].reshape(-1)[i] += h
            pm[k].reshape(-1)[i] -= h
            fd = (L(pp) - L(pm)) / (2 * h)
            g = grads[k].reshape(-1)[i]
            assert abs(fd - g) <= 1e-6 * max(1.0, abs(g)) + 1e-8, (k, int(i), fd, g)
        assert np.abs(grads[k]).max() > 0, k


def test_cls_bf16_mode_stays_within_rounding_of_exact():
    cfg = tiny_bert("bf16", d_model=64, head_dim=32, hsm_m1=96, hsm_m2=160)
    W, s_i, s_prev, inertia, s_fin, lab = setup_cls(cfg, n=12, n_cls=4, std=0.05)
    l64, g64, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, s_fin, lab, 1.0, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    l16, g16, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, s_fin, lab, 1.0, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1,
                                           bf16=True)
    assert abs(l16 - l64) <= 1e-2 * abs(l64)
    for k in HT.HSM_PARAMS:
        e = np.linalg.norm(g16[k] - g64[k]) / np.linalg.norm(g64[k])
        assert e < 3e-2, (k, e)


def test_one_class_task_term_vanishes():
    """With a single class the softmax is 1 whatever the logits: the task term and its gradient
    are exactly zero, so the step equals the similarity-only step."""
    cfg = tiny_bert(n_classes=1)
    W, s_i, s_prev, inertia, s_fin, _ = setup_cls(cfg, n=5, n_cls=3)
    lab = torch.zeros(3, dtype=torch.long)
    l1, g1, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, s_fin, lab, 2.0, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    l0, g0, _, _ = HT.hsm_cls_train_step(W, cfg, s_i, s_prev, inertia, s_fin, [], 2.0, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    assert l1 == l0
    for k in HT.HSM_PARAMS:
        np.testing.assert_array_equal(g1[k], g0[k])
