"""GPU parity of the HSM training step (Sec. 4.2; Sec. 5.1 "Training"; App. D) through the C
ABI against the training oracle on the same seeded examples: the loss, every parameter's
gradient, the AdamW moments and the updated parameters, over one and several steps; the
inference path after training; device-side validation of the targets.

Tolerances: norm-wise relative error per parameter tensor within the precision contract
(1e-4 fp32, 2e-2 bf16); the oracle rounds GEMM inputs to bf16 where the bf16 models do."""
import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from oracle import hsm_train as HT
from parity_utils import Pair, compare_prefill, TOL

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


def cfg_of(family, dtype, **kw):
    base = dict(family=family, n_layers=4, d_model=128, n_heads=2, head_dim=64, d_ffn=256, vocab=1000, max_pos=64,
                dtype=dtype, max_batch=2, max_seq=64, hsm_m1=256, hsm_m2=512)
    base.update(kw)
    return synth.ModelConfig(**base)


def rel(a, b):
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30)


def oracle_run(W, cfg, batch, steps, lr, b1, b2, eps, wd):
    s_i, s_prev, inertia, tgt = batch
    bf = cfg.dtype == "bf16"
    params, state, out = None, None, []
    for t in range(1, steps + 1):
        loss, grads, params, state = HT.hsm_train_step(W, cfg, s_i.double(), s_prev.double(), inertia.double(),
                                                       tgt.long(), lr, b1, b2, eps, wd, t, params=params,
                                                       state=state, bf16=bf)
        out.append((loss, grads, params, state))
    return out


def adam_eps_for(W, cfg, batch):
    """An AdamW eps at the median gradient magnitude, so that the first update is a smooth
    function of the gradient (with eps far below it the update is lr * sign(g))."""
    g = oracle_run(W, cfg, batch, 1, 1e-3, 0.9, 0.999, 1e-8, 0.0)[0][1]
    return float(np.median(np.abs(np.concatenate([v.ravel() for v in g.values()]))))


def gpu_run(model, cfg, batch, steps, lr, b1, b2, eps, wd, cap=None):
    s_i, s_prev, inertia, tgt = [x.cuda() for x in batch]
    n = s_i.shape[0]
    adept.adept_hsm_train_init(model.h, cap or n)
    theta0 = [model.hsm_train_read(adept.HSM_PARAMS, p).cpu().numpy() for p in range(13)]
    loss = torch.zeros(1, device="cuda")
    out = []
    for _ in range(steps):
        adept.adept_hsm_train_step(model.h, n, s_i, s_prev, inertia, tgt, lr, b1, b2, eps, wd, loss_out=loss)
        model.check()
        rd = lambda what: {adept.HSM_PARAM_NAMES[p]: model.hsm_train_read(what, p).cpu().numpy() for p in range(13)}
        out.append((float(loss.item()), rd(adept.HSM_GRADS), rd(adept.HSM_PARAMS), rd(adept.HSM_MOMENT1),
                    rd(adept.HSM_MOMENT2)))
    return theta0, out


def check_step(cfg, W, o, g, theta0_o, tol, what):
    loss_o, grads_o, params_o, state_o = o
    loss_g, grads_g, params_g, m1_g, m2_g = g
    assert abs(loss_g - loss_o) <= max(tol * 0.1, 1e-6) * abs(loss_o), f"{what}: loss {loss_g} vs {loss_o}"
    for k in HT.HSM_PARAMS:
        shp = params_o[k].shape
        e = rel(grads_g[k], grads_o[k])
        assert e <= tol, f"{what}: gradient of {k}: {e:.3e}"
        e = rel(m1_g[k], state_o[k][0])
        assert e <= tol, f"{what}: first moment of {k}: {e:.3e}"
        e = rel(m2_g[k], state_o[k][1])
        assert e <= 2 * tol, f"{what}: second moment of {k}: {e:.3e}"
        # the update itself, relative to its own size
        e = rel(params_g[k].reshape(shp) - theta0_o[k], params_o[k] - theta0_o[k])
        assert e <= tol, f"{what}: update of {k}: {e:.3e}"


@pytest.mark.parametrize("family,dtype,n,vocab", [(synth.LLAMA, "f32", 13, 1000), (synth.GPT2, "f32", 8, 1000),
                                                  (synth.LLAMA, "bf16", 13, 1000), (synth.GPT2, "bf16", 37, 1000),
                                                  (synth.GPT2, "bf16", 1, 1000), (synth.LLAMA, "bf16", 45, 4099)])
def test_one_step_matches_oracle(family, dtype, n, vocab):
    """Loss, gradients, moments and update of one step (n examples; ragged n exercises the
    padded transposes; n <= 16 takes the generation-step GEMM for the n-row products; a
    4099-token vocabulary splits the head's input-gradient product over K and pads its rows)."""
    cfg = cfg_of(family, dtype, vocab=vocab)
    W = synth.make_weights(cfg, seed=3, std=0.05, gain_std=0.1 if dtype == "f32" else None)
    batch = synth.hsm_train_batch(cfg, n, seed=5)
    eps = adam_eps_for(W, cfg, batch)
    o = oracle_run(W, cfg, batch, 1, 1e-3, 0.9, 0.999, eps, 0.01)
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    m = adept.Model(cfg, W)
    try:
        theta0, g = gpu_run(m, cfg, batch, 1, 1e-3, 0.9, 0.999, eps, 0.01, cap=n + 5)
        for p, k in enumerate(adept.HSM_PARAM_NAMES):
            np.testing.assert_array_equal(theta0[p], W[k].float().numpy().ravel())
        check_step(cfg, W, o[0], g[0], theta0_o, TOL[dtype], f"{dtype} n={n}")
    finally:
        m.close()


@pytest.mark.parametrize("family,dtype", [(synth.LLAMA, "f32"), (synth.GPT2, "bf16")])
def test_three_steps_match_oracle(family, dtype):
    """Three steps on one batch: each step's forward uses the weights the previous update
    wrote back (bf16 copies for the products, transposed copies for the input gradients)."""
    cfg = cfg_of(family, dtype)
    W = synth.make_weights(cfg, seed=4, std=0.05, gain_std=0.1 if dtype == "f32" else None)
    batch = synth.hsm_train_batch(cfg, 24, seed=6)
    eps = adam_eps_for(W, cfg, batch)
    o = oracle_run(W, cfg, batch, 3, 3e-3, 0.8, 0.95, eps, 0.0)
    m = adept.Model(cfg, W)
    try:
        _, g = gpu_run(m, cfg, batch, 3, 3e-3, 0.8, 0.95, eps, 0.0)
    finally:
        m.close()
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    for t in range(3):
        # updates compared cumulatively, from the initial parameters
        check_step(cfg, W, o[t], g[t], theta0_o, TOL[dtype], f"step {t + 1}")
    assert o[2][0] < o[0][0]


def test_inference_uses_the_trained_hsm():
    """After two steps the model's prompt pass maps exiting tokens with the trained HSM:
    forced-exit prefill against the inference oracle built from the oracle's updated
    parameters (matrices rounded to bf16 as the device stores them)."""
    cfg = cfg_of(synth.GPT2, "bf16", max_batch=2, max_seq=40)
    W = synth.make_weights(cfg, seed=8, std=0.05)
    batch = synth.hsm_train_batch(cfg, 16, seed=9)
    eps = adam_eps_for(W, cfg, batch)
    o = oracle_run(W, cfg, batch, 2, 1e-2, 0.9, 0.999, eps, 0.0)
    pair = Pair(cfg, weights=W)
    try:
        gpu_run(pair.gm, cfg, batch, 2, 1e-2, 0.9, 0.999, eps, 0.0)
        W2 = dict(W)
        for k, v in o[1][2].items():
            t = torch.as_tensor(v)
            W2[k] = t.to(torch.bfloat16) if t.dim() == 2 and k != "hsm.conv_w" else t.to(torch.float64)
        pair.om = O.OracleModel(cfg, W2)
        B, P = 2, 30
        tokens = synth.randint(10, "train-prompt", B * P, 0, cfg.vocab - 1).numpy().reshape(B, P)
        forced = synth.forced_exits_uniform(11, B * P, 2, cfg.n_layers).numpy().reshape(B, P)
        compare_prefill(pair, tokens, 0.5, forced=forced)
    finally:
        pair.close()


def test_bad_target_flags_device_input_and_drops_the_row():
    """A target outside [0, vocab) is flagged (DEVICE_INPUT at the status check); its row adds
    nothing to the loss or the gradients: the loss is the others' sum over n."""
    cfg = cfg_of(synth.LLAMA, "f32")
    W = synth.make_weights(cfg, seed=2, std=0.05, gain_std=0.1)
    s_i, s_prev, inertia, tgt = synth.hsm_train_batch(cfg, 6, seed=3)
    bad = tgt.clone()
    bad[4] = cfg.vocab
    keep = [0, 1, 2, 3, 5]
    o = HT.hsm_train_step(W, cfg, s_i[keep].double(), s_prev[keep].double(), inertia[keep].double(), tgt[keep].long(),
                          1e-3, 0.9, 0.999, 1e-8, 0.0, 1)
    m = adept.Model(cfg, W)
    try:
        adept.adept_hsm_train_init(m.h, 6)
        loss = torch.zeros(1, device="cuda")
        adept.adept_hsm_train_step(m.h, 6, s_i.cuda(), s_prev.cuda(), inertia.cuda(), bad.cuda(), 1e-3,
                                   loss_out=loss)
        with pytest.raises(adept.AdeptError) as ei:
            m.check()
        assert ei.value.status == 6
        assert abs(loss.item() - o[0] * 5 / 6) <= 1e-5 * abs(o[0])
        g = m.hsm_train_read(adept.HSM_GRADS, 3).cpu().numpy()      # fc1_w
        assert rel(g, o[1]["hsm.fc1_w"].ravel() * 5 / 6) <= TOL["f32"]
        with pytest.raises(adept.AdeptError):
            adept.adept_hsm_train_step(m.h, 7, s_i.cuda(), s_prev.cuda(), inertia.cuda(), tgt.cuda(), 1e-3)
    finally:
        m.close()


def test_gpt2_small_shape_step_matches_oracle():
    """GPT-2-small shapes (D 768, HSM widths 3072 / 6144, vocabulary 50257, bf16), 48 examples:
    one step's loss, gradients and update against the oracle."""
    cfg = synth.gpt2_small_config(n_layers=2, max_batch=1, max_seq=16)
    W = synth.make_weights(cfg, seed=1)
    batch = synth.hsm_train_batch(cfg, 48, seed=2)
    eps = 1e-6
    o = oracle_run(W, cfg, batch, 1, 1e-4, 0.9, 0.999, eps, 0.0)
    theta0_o = {k: W[k].double().numpy() for k in HT.HSM_PARAMS}
    m = adept.Model(cfg, W)
    try:
        _, g = gpu_run(m, cfg, batch, 1, 1e-4, 0.9, 0.999, eps, 0.0)
    finally:
        m.close()
    loss_o, grads_o, params_o, _ = o[0]
    loss_g, grads_g, params_g, _, _ = g[0]
    assert abs(loss_g - loss_o) <= 1e-3 * loss_o
    for k in HT.HSM_PARAMS:
        assert rel(grads_g[k], grads_o[k]) <= TOL["bf16"], k
        # eps far below the gradients: the update is lr * sign(g) almost everywhere; the
        # elements whose sign differs are those with gradients near zero
        du_g = params_g[k].reshape(params_o[k].shape) - theta0_o[k]
        du_o = params_o[k] - theta0_o[k]
        assert np.mean(np.sign(du_g) != np.sign(du_o)) <= 0.02, k
