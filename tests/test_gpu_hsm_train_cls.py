"""GPU parity of the encoder (classification) HSM training step (Sec. 4.3) through the C ABI
against the training oracle on the same seeded examples: similarity loss against the
original final states plus the frozen pooler + classifier's cross-entropy on the labelled
rows; the loss, every parameter's gradient, the AdamW moments and the update, over one and
several steps; the encoder's prompt pass after training; device-side label validation and
the argument checks.

Tolerances: norm-wise relative error per parameter tensor within the precision contract
(1e-4 fp32, 2e-2 bf16); the oracle rounds GEMM inputs to bf16 where the bf16 models do."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import adept_oracle as O
from oracle import hsm_train as HT
from parity_utils import Pair, compare_prefill, TOL
from test_gpu_hsm_train import check_step, rel

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


def enc_cfg(dtype, **kw):
    base = dict(family=synth.BERT, n_layers=4, d_model=128, n_heads=2, head_dim=64, d_ffn=256, vocab=1000, max_pos=64,
                n_classes=2, dtype=dtype, norm_eps=1e-12, max_batch=2, max_seq=64, hsm_m1=256, hsm_m2=512)
    base.update(kw)
    return synth.ModelConfig(**base)


def oracle_run(W, cfg, batch, steps, w, lr, b1, b2, eps, wd):
    s_i, s_prev, inertia, s_fin, lab = batch
    params, state, out = None, None, []
    for t in range(1, steps + 1):
        loss, grads, params, state = HT.hsm_cls_train_step(W, cfg, s_i.double(), s_prev.double(), inertia.double(),
                                                           s_fin.double(), lab.long(), w, lr, b1, b2, eps, wd, t,
                                                           params=params, state=state, bf16=cfg.dtype == "bf16")
        out.append((loss, grads, params, state))
    return out


def adam_eps_for(W, cfg, batch, w):
    g = oracle_run(W, cfg, batch, 1, w, 1e-3, 0.9, 0.999, 1e-8, 0.0)[0][1]
    return float(np.median(np.abs(np.concatenate([v.ravel() for v in g.values()]))))


def gpu_run(model, batch, steps, w, lr, b1, b2, eps, wd, cap=None):
    s_i, s_prev, inertia, s_fin, lab = [x.cuda() for x in batch]
    n = s_i.shape[0]
    adept.adept_hsm_train_init(model.h, cap or n)
    theta0 = [model.hsm_train_read(adept.HSM_PARAMS, p).cpu().numpy() for p in range(13)]
    loss = torch.zeros(1, device="cuda")
    out = []
    for _ in range(steps):
        adept.adept_hsm_train_step_cls(model.h, n, s_i, s_prev, inertia, s_fin, lab if lab.numel() else None, lr,
                                       cls_weight=w, beta1=b1, beta2=b2, eps=eps, weight_decay=wd, loss_out=loss)
        model.check()
        rd = lambda what: {adept.HSM_PARAM_NAMES[p]: model.hsm_train_read(what, p).cpu().numpy() for p in range(13)}
        out.append((float(loss.item()), rd(adept.HSM_GRADS), rd(adept.HSM_PARAMS), rd(adept.HSM_MOMENT1),
                    rd(adept.HSM_MOMENT2)))
    return theta0, out


@pytest.mark.parametrize("dtype,n,n_cls,n_classes,w", [("f32", 13, 4, 2, 1.0), ("bf16", 37, 5, 2, 1.0),
                                                        ("bf16", 1, 1, 2, 1.0), ("bf16", 20, 0, 2, 1.0),
                                                        ("bf16", 9, 9, 3, 0.5), ("f32", 150, 17, 5, 2.0)])
def test_one_step_matches_oracle(dtype, n, n_cls, n_classes, w):
    """Loss, gradients, moments and update of one step (no labelled rows, some, all; two to
    five classes; a single example; 150 rows span two GEMM row tiles with a ragged tail)."""
    cfg = enc_cfg(dtype, n_classes=n_classes)
    W = synth.make_weights(cfg, seed=3, std=0.05, gain_std=0.1 if dtype == "f32" else None)
    batch = synth.hsm_cls_batch(cfg, n, n_cls, seed=5)
    eps = adam_eps_for(W, cfg, batch, w)
    o = oracle_run(W, cfg, batch, 1, w, 1e-3, 0.9, 0.999, eps, 0.01)
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    m = adept.Model(cfg, W)
    try:
        _, g = gpu_run(m, batch, 1, w, 1e-3, 0.9, 0.999, eps, 0.01, cap=n + 3)
        check_step(cfg, W, o[0], g[0], theta0_o, TOL[dtype], f"{dtype} n={n} n_cls={n_cls}")
    finally:
        m.close()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_three_steps_match_oracle(dtype):
    """Three steps on one batch, each forward on the weights the previous update wrote back."""
    cfg = enc_cfg(dtype)
    W = synth.make_weights(cfg, seed=4, std=0.05, gain_std=0.1 if dtype == "f32" else None)
    batch = synth.hsm_cls_batch(cfg, 24, 6, seed=6)
    eps = adam_eps_for(W, cfg, batch, 1.0)
    o = oracle_run(W, cfg, batch, 3, 1.0, 3e-3, 0.8, 0.95, eps, 0.0)
    m = adept.Model(cfg, W)
    try:
        _, g = gpu_run(m, batch, 3, 1.0, 3e-3, 0.8, 0.95, eps, 0.0)
    finally:
        m.close()
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    check_steps(o, g, theta0_o, 0.8, 0.95, TOL[dtype])
    assert o[2][0] < o[0][0]


def check_steps(o, g, theta0_o, b1, b2, tol):
    """Several steps, each error against the size of what it sums rather than the sum: the
    first moment against b1 |m_prev| + (1 - b1) |g| and the parameters against the path length
    sum_t |update_t| (a gradient that changes sign between steps cancels in m and in the
    cumulative update; a scalar such as the convolution bias then has no relative scale)."""
    prev_m = {k: np.zeros_like(theta0_o[k]) for k in HT.HSM_PARAMS}
    prev_p = dict(theta0_o)
    path = {k: 0.0 for k in HT.HSM_PARAMS}
    for t, (ot, gt) in enumerate(zip(o, g)):
        loss_o, grads_o, params_o, state_o = ot
        loss_g, grads_g, params_g, m1_g, m2_g = gt
        what = f"step {t + 1}"
        assert abs(loss_g - loss_o) <= max(tol * 0.1, 1e-6) * abs(loss_o), f"{what}: loss {loss_g} vs {loss_o}"
        for k in HT.HSM_PARAMS:
            shp = params_o[k].shape
            assert rel(grads_g[k], grads_o[k]) <= tol, f"{what}: gradient of {k}"
            den = np.linalg.norm(b1 * np.abs(prev_m[k]) + (1 - b1) * np.abs(grads_o[k]))
            assert np.linalg.norm(m1_g[k].reshape(shp) - state_o[k][0]) <= tol * den, f"{what}: first moment of {k}"
            assert rel(m2_g[k], state_o[k][1]) <= 2 * tol, f"{what}: second moment of {k}"
            path[k] += np.linalg.norm(params_o[k] - prev_p[k])
            assert np.linalg.norm(params_g[k].reshape(shp) - params_o[k]) <= tol * path[k], f"{what}: update of {k}"
            prev_m[k], prev_p[k] = state_o[k][0], params_o[k]


def test_encoder_prompt_pass_uses_the_trained_hsm():
    """After two steps the encoder's forced-exit prompt pass (final states and class logits)
    matches the inference oracle built from the oracle's updated parameters."""
    cfg = enc_cfg("bf16", max_batch=2, max_seq=40)
    W = synth.make_weights(cfg, seed=8, std=0.05)
    batch = synth.hsm_cls_batch(cfg, 16, 4, seed=9)
    eps = adam_eps_for(W, cfg, batch, 1.0)
    o = oracle_run(W, cfg, batch, 2, 1.0, 1e-2, 0.9, 0.999, eps, 0.0)
    pair = Pair(cfg, weights=W)
    try:
        gpu_run(pair.gm, batch, 2, 1.0, 1e-2, 0.9, 0.999, eps, 0.0)
        W2 = dict(W)
        for k, v in o[1][2].items():
            t = torch.as_tensor(v)
            W2[k] = t.to(torch.bfloat16) if t.dim() == 2 and k != "hsm.conv_w" else t.to(torch.float64)
        pair.om = O.OracleModel(cfg, W2)
        B, P = 2, 30
        tokens = synth.randint(10, "train-prompt", B * P, 0, cfg.vocab - 1).numpy().reshape(B, P)
        forced = synth.forced_exits_uniform(11, B * P, 2, cfg.n_layers).numpy().reshape(B, P)
        compare_prefill(pair, tokens, 0.5, forced=forced, check_cache=False)
    finally:
        pair.close()


def test_bad_label_flags_device_input_and_drops_the_row():
    """A label outside [0, n_classes) is flagged (DEVICE_INPUT at the status check); its row
    adds no task loss: loss = similarity + w / n_cls * (the other rows' cross-entropy)."""
    cfg = enc_cfg("f32")
    W = synth.make_weights(cfg, seed=2, std=0.05, gain_std=0.1)
    s_i, s_prev, inertia, s_fin, lab = synth.hsm_cls_batch(cfg, 8, 4, seed=3)
    bad = lab.clone()
    bad[2] = cfg.n_classes
    p = {k: W[k].double() for k in HT.HSM_PARAMS}
    with torch.no_grad():
        st = HT.hsm_forward(p, cfg, s_i.double(), s_prev.double(), inertia.double())
        sim = float(torch.mean(1.0 - HT.cosine_rows(st, s_fin.double())))
        ce = F.cross_entropy(HT.cls_head_logits(W, cfg, st[:4]), lab.long(), reduction="none").numpy()
    want = sim + 0.8 / 4 * (ce.sum() - ce[2])
    m = adept.Model(cfg, W)
    try:
        adept.adept_hsm_train_init(m.h, 8)
        loss = torch.zeros(1, device="cuda")
        adept.adept_hsm_train_step_cls(m.h, 8, s_i.cuda(), s_prev.cuda(), inertia.cuda(), s_fin.cuda(), bad.cuda(),
                                       1e-3, cls_weight=0.8, loss_out=loss)
        with pytest.raises(adept.AdeptError) as ei:
            m.check()
        assert ei.value.status == 6
        assert abs(loss.item() - want) <= 1e-5 * abs(want)
    finally:
        m.close()


def test_argument_checks():
    """The encoder step refuses decoders, n_cls above n, a negative weight; the decoder step
    refuses encoders."""
    ecfg = enc_cfg("f32")
    W = synth.make_weights(ecfg, seed=2, std=0.05)
    s_i, s_prev, inertia, s_fin, lab = [x.cuda() for x in synth.hsm_cls_batch(ecfg, 4, 2, seed=3)]
    m = adept.Model(ecfg, W)
    try:
        adept.adept_hsm_train_init(m.h, 4)
        with pytest.raises(adept.AdeptError):
            adept.adept_hsm_train_step(m.h, 4, s_i, s_prev, inertia, lab, 1e-3)
        with pytest.raises(adept.AdeptError):
            adept.adept_hsm_train_step_cls(m.h, 1, s_i, s_prev, inertia, s_fin, lab, 1e-3)
        with pytest.raises(adept.AdeptError):
            adept.adept_hsm_train_step_cls(m.h, 4, s_i, s_prev, inertia, s_fin, lab, 1e-3, cls_weight=-1.0)
        adept.adept_hsm_train_step_cls(m.h, 4, s_i, s_prev, inertia, s_fin, lab, 1e-3)
        m.check()
    finally:
        m.close()
    dcfg = synth.ModelConfig(**{**ecfg.__dict__, "family": synth.GPT2, "n_classes": 0, "norm_eps": 1e-5})
    Wd = synth.make_weights(dcfg, seed=2, std=0.05)
    md = adept.Model(dcfg, Wd)
    try:
        adept.adept_hsm_train_init(md.h, 4)
        with pytest.raises(adept.AdeptError):
            adept.adept_hsm_train_step_cls(md.h, 4, s_i, s_prev, inertia, s_fin, lab, 1e-3)
    finally:
        md.close()


def test_bert_base_shape_step_matches_oracle():
    """BERT-base shapes (D 768, HSM widths 3072 / 6144, two classes, bf16), 48 examples of
    which 6 labelled: one step's loss, gradients and update signs against the oracle."""
    cfg = synth.bert_base_config(n_layers=2, max_batch=1, max_seq=16)
    W = synth.make_weights(cfg, seed=1)
    batch = synth.hsm_cls_batch(cfg, 48, 6, seed=2)
    o = oracle_run(W, cfg, batch, 1, 1.0, 1e-4, 0.9, 0.999, 1e-6, 0.0)
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    m = adept.Model(cfg, W)
    try:
        _, g = gpu_run(m, batch, 1, 1.0, 1e-4, 0.9, 0.999, 1e-6, 0.0)
    finally:
        m.close()
    loss_o, grads_o, params_o, _ = o[0]
    loss_g, grads_g, params_g, _, _ = g[0]
    assert abs(loss_g - loss_o) <= 1e-3 * loss_o
    for k in HT.HSM_PARAMS:
        assert rel(grads_g[k], grads_o[k]) <= TOL["bf16"], k
        du_g = params_g[k].reshape(params_o[k].shape) - theta0_o[k]
        du_o = params_o[k] - theta0_o[k]
        assert np.mean(np.sign(du_g) != np.sign(du_o)) <= 0.02, k
