"""The persistent generation-step launch (FUSED_DECODE) against the multi-launch step on
the same weights and inputs, and against the oracle.  Forced exits make the two device
paths take identical decisions, so exit layers, greedy tokens (outside ties) and every
KV entry written by a layer or a skipped-layer fill are compared; logits and final
states within the bf16 row tolerance."""
import numpy as np
import pytest
import torch

import synth
from parity_utils import TOL, Pair, assert_rows_close, compare_decode, compare_prefill, row_rel_err

import paper_2601_03700_gb300 as adept

# The persistent step showed an intermittent device fault on Llama-7B-shaped models whose
# cause is not yet found; it is not run on a GPU until it is (it is off by default and the
# library takes the multi-launch step).
pytestmark = [pytest.mark.gpu, pytest.mark.skip(reason="persistent generation step disabled pending a fault investigation")]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


def small(family, **kw):
    base = dict(family=family, n_layers=6, d_model=256, n_heads=4, head_dim=64, d_ffn=512, vocab=1000,
                max_pos=200, n_classes=0, dtype="bf16", max_batch=4, max_seq=200, hsm_m1=512, hsm_m2=1024)
    base.update(kw)
    return synth.ModelConfig(**base)


def _run(cfg, W, fused, B, P, steps, seed, delta=0.5, step_forced=True, identity=False):
    m = adept.Model(cfg, W)
    adept.adept_set_option(m.h, adept.OPT_FUSED_DECODE, fused)
    if identity:
        adept.adept_set_option(m.h, adept.OPT_HSM_IDENTITY, 1)
    if fused:
        assert m.fused_decode_batch() >= B, m.fused_decode_reason()
    N = cfg.n_layers
    tokens = synth.make_tokens(seed, B, P, cfg.vocab).cuda()
    pf = synth.forced_exits_uniform(seed, B * P, 2, N).view(B, P).cuda()
    ex, lg, nx, _ = m.prefill(tokens, delta, pf)
    fs = synth.forced_exits_uniform(seed + 1, steps * B, 2, N).view(steps, B).cuda()
    out = []
    for s in range(steps):
        ex, lg, nx, sim = m.decode_step(nx, delta, fs[s] if step_forced else None)
        out.append(dict(ex=ex.cpu(), lg=lg.cpu(), nx=nx.cpu(), sim=sim.cpu(), fin=m.final_states(B).cpu()))
    m.check()
    kv = {}
    for layer in range(1, N + 1):
        for b in range(B):
            k, v = m.read_kv(layer, b, 0, P + steps)
            kv[(layer, b)] = (k.float().cpu(), v.float().cpu())
    m.close()
    return out, kv


def _compare(a, b, tol):
    for s, (x, y) in enumerate(zip(a[0], b[0])):
        assert torch.equal(x["ex"], y["ex"]), f"step {s} exit layers"
        assert_rows_close(x["lg"].numpy(), y["lg"].numpy().astype(np.float64), tol, f"step {s} logits")
        assert_rows_close(x["fin"].numpy(), y["fin"].numpy().astype(np.float64), tol, f"step {s} final states")
        lg = y["lg"].numpy()
        top2 = np.sort(lg, axis=1)[:, -2:]
        clear = (top2[:, 1] - top2[:, 0]) > tol * np.abs(top2[:, 1]).clip(1.0)
        assert np.array_equal(x["nx"].numpy()[clear], y["nx"].numpy()[clear]), f"step {s} greedy tokens"
    for key in a[1]:
        for t in range(2):
            ka, kb = a[1][key][t].reshape(a[1][key][t].shape[0], -1), b[1][key][t].reshape(b[1][key][t].shape[0], -1)
            assert_rows_close(ka.numpy(), kb.numpy().astype(np.float64), tol, f"cache {key} {'kv'[t]}")


@pytest.mark.parametrize("family,kw", [(synth.LLAMA, dict(n_heads=2, head_dim=128)),
                                       (synth.LLAMA, dict(n_heads=4, n_kv_heads=2, head_dim=64)),
                                       (synth.GPT2, {})])
def test_fused_step_matches_multi_launch_step(family, kw):
    cfg = small(family, **kw)
    W = synth.make_weights(cfg, seed=31)
    a = _run(cfg, W, 1, 3, 70, 6, seed=31)
    b = _run(cfg, W, 0, 3, 70, 6, seed=31)
    _compare(a, b, TOL["bf16"])


def test_fused_step_hsm_identity_and_batch_of_one():
    cfg = small(synth.LLAMA, n_layers=8, n_heads=2, head_dim=128)
    W = synth.make_weights(cfg, seed=32)
    a = _run(cfg, W, 1, 1, 33, 5, seed=32, identity=True)
    b = _run(cfg, W, 0, 1, 33, 5, seed=32, identity=True)
    _compare(a, b, TOL["bf16"])


def test_fused_step_every_token_leaves_at_layer_two():
    """All rows exit at the first eligible layer: the layer loop ends early, every
    skipped layer 3..N is filled from s~, and the head reads only mapped states."""
    cfg = small(synth.GPT2, n_layers=6)
    W = synth.make_weights(cfg, seed=33)
    res = []
    for fused in (1, 0):
        m = adept.Model(cfg, W)
        adept.adept_set_option(m.h, adept.OPT_FUSED_DECODE, fused)
        tokens = synth.make_tokens(33, 4, 20, cfg.vocab).cuda()
        ex, lg, nx, _ = m.prefill(tokens, 0.5, torch.full((4, 20), 2, dtype=torch.int32, device="cuda"))
        steps = []
        for s in range(3):
            ex, lg, nx, sim = m.decode_step(nx, 0.5, torch.full((4,), 2, dtype=torch.int32, device="cuda"))
            steps.append((ex.cpu(), lg.cpu(), nx.cpu()))
            assert torch.all(ex.cpu() == 2)
        m.check()
        kv = [m.read_kv(r, b, 20, 3)[0].float().cpu() for r in range(1, 7) for b in range(4)]
        res.append((steps, kv))
        m.close()
    for (ea, la, na), (eb, lb, nb) in zip(res[0][0], res[1][0]):
        assert torch.equal(ea, eb)
        assert row_rel_err(la.numpy(), lb.numpy().astype(np.float64)).max() < TOL["bf16"]
    for x, y in zip(res[0][1], res[1][1]):
        assert row_rel_err(x.reshape(3, -1).numpy(), y.reshape(3, -1).numpy().astype(np.float64)).max() < TOL["bf16"]


def test_fused_step_is_deterministic():
    cfg = small(synth.LLAMA, n_heads=4, head_dim=64)
    W = synth.make_weights(cfg, seed=34)
    a = _run(cfg, W, 1, 4, 40, 4, seed=34, step_forced=False)
    b = _run(cfg, W, 1, 4, 40, 4, seed=34, step_forced=False)
    for x, y in zip(a[0], b[0]):
        for k in ("ex", "lg", "nx", "fin"):
            assert torch.equal(x[k], y[k]), k
        assert torch.equal(x["sim"].nan_to_num(7.0), y["sim"].nan_to_num(7.0))
    for key in a[1]:
        assert torch.equal(a[1][key][0], b[1][key][0]) and torch.equal(a[1][key][1], b[1][key][1])


@pytest.mark.parametrize("family", [synth.LLAMA, synth.GPT2])
def test_fused_step_against_oracle_threshold(family):
    """The fused step against the oracle in threshold mode (teacher-forced tokens; band
    tokens re-run with the oracle's decisions)."""
    cfg = small(family, n_layers=5)
    pair = Pair(cfg, seed=35, std=0.05)
    adept.adept_set_option(pair.gm.h, adept.OPT_FUSED_DECODE, 1)
    assert pair.gm.fused_decode_batch() >= 2, pair.gm.fused_decode_reason()
    tokens = synth.make_tokens(35, 2, 48, cfg.vocab).numpy()
    ores, cache, g = compare_prefill(pair, tokens, 0.8)
    compare_decode(pair, cache, ores.next_token, 4, 0.8)
    pair.compare_cache(cache, 2, 52)
    pair.close()
