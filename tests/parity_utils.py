"""Helpers shared by the GPU parity tests: run the CUDA library and the CPU oracle on the
same seeded inputs and compare them under the tolerances of the precision contract."""
from __future__ import annotations

import numpy as np
import torch

import synth
import paper_2601_03700_gb300 as adept
from oracle import adept_oracle as O

# norm-wise relative error per row (hidden states, logits, KV entries)
TOL = {"f32": 1e-4, "bf16": 2e-2}
BAND = 1e-3          # similarity band around delta inside which the oracle's decision is taken


def row_rel_err(got: np.ndarray, want: np.ndarray) -> np.ndarray:
    got = np.asarray(got, dtype=np.float64).reshape(len(want), -1)
    want = np.asarray(want, dtype=np.float64).reshape(len(want), -1)
    num = np.linalg.norm(got - want, axis=1)
    den = np.maximum(np.linalg.norm(want, axis=1), 1e-30)
    return num / den


def assert_rows_close(got, want, tol, what):
    e = row_rel_err(got, want)
    worst = int(np.argmax(e)) if len(e) else 0
    assert len(e) == 0 or e.max() <= tol, f"{what}: max row rel err {e.max():.3e} at row {worst} (tol {tol})"
    return float(e.max()) if len(e) else 0.0


class Pair:
    """A library model and an oracle model built from the same synthetic weights."""

    def __init__(self, cfg: synth.ModelConfig, seed: int = 0, weights=None, std: float = 0.02):
        self.cfg = cfg
        self.W = weights if weights is not None else synth.make_weights(cfg, seed=seed, std=std)
        self.om = O.OracleModel(cfg, self.W)
        self.gm = adept.Model(cfg, self.W)
        self.tol = TOL[cfg.dtype]
        self.cross = None   # encoder-decoder decoders: the oracle's O.CrossSource

    def close(self):
        self.gm.close()

    def gpu_kv(self, layer, seq, n_pos):
        k, v = self.gm.read_kv(layer, seq, 0, n_pos)
        return k.float().cpu().numpy(), v.float().cpu().numpy()

    def compare_cache(self, cache: O.OracleCache, batch: int, n_pos: int):
        worst = 0.0
        for l in range(1, self.cfg.n_layers + 1):
            for b in range(batch):
                k, v = self.gpu_kv(l, b, n_pos)
                worst = max(worst, assert_rows_close(k, cache.K[l - 1][b, :n_pos], self.tol, f"K layer {l} seq {b}"))
                worst = max(worst, assert_rows_close(v, cache.V[l - 1][b, :n_pos], self.tol, f"V layer {l} seq {b}"))
        return worst


def band_tokens(sim: np.ndarray, delta: float) -> np.ndarray:
    """Tokens with any tested similarity within BAND of delta."""
    with np.errstate(invalid="ignore"):
        close = np.abs(sim - delta) <= BAND
    return np.any(close & ~np.isnan(sim), axis=1)


def decisions_agree_outside_band(g_sim: np.ndarray, o_sim: np.ndarray, delta: float, o_exit: np.ndarray):
    """At every layer the oracle tested, the GPU's own similarity decides the same way
    wherever the oracle's similarity is outside the band."""
    tested = ~np.isnan(o_sim)
    assert np.array_equal(tested, ~np.isnan(g_sim)), "tested layers differ"
    with np.errstate(invalid="ignore"):
        outside = tested & (np.abs(o_sim - delta) > BAND)
        gd = g_sim >= delta
        od = o_sim >= delta
    bad = outside & (gd != od)
    assert not bad.any(), f"{int(bad.sum())} decisions differ outside the band"


def run_prefill(pair: Pair, tokens: np.ndarray, delta: float, forced=None, hsm_identity=False, metric="global",
                all_at_once=False, stop_entirely=False):
    """Returns (oracle result, oracle cache, gpu outputs dict); in threshold mode with band
    tokens, the GPU is re-run with the oracle's exit layers forced.  metric / all_at_once:
    the exit-rule variant (the device options are set here too)."""
    cfg = pair.cfg
    B, P = tokens.shape
    cache = O.OracleCache(cfg, cfg.max_batch, cfg.max_seq)
    ores = O.prefill(pair.om, cache, tokens, delta, forced, hsm_mode="identity" if hsm_identity else "hsm",
                     metric=metric, all_at_once=all_at_once, stop_entirely=stop_entirely, cross=pair.cross)
    if cfg.family == synth.BERT:
        adept.adept_set_option(pair.gm.h, adept.OPT_STOP_ENTIRELY, int(stop_entirely))
    adept.adept_set_option(pair.gm.h, adept.OPT_EXIT_METRIC, {"global": 0, "local": 1, "both": 2}[metric])
    adept.adept_set_option(pair.gm.h, adept.OPT_ALL_AT_ONCE, int(all_at_once))
    adept.adept_set_option(pair.gm.h, adept.OPT_HSM_IDENTITY, int(hsm_identity))
    tk = torch.as_tensor(tokens, dtype=torch.int32, device="cuda")
    fz = None if forced is None else torch.as_tensor(np.asarray(forced).reshape(B, P), dtype=torch.int32, device="cuda")
    ex, lg, nx, sim = pair.gm.prefill(tk, delta, fz)
    pair.gm.check()
    g_exit = ex.cpu().numpy()
    g_sim = sim.cpu().numpy()
    forced_rerun = False
    if forced is None:
        band = band_tokens(ores.sim, delta)
        if band.any():
            forced_rerun = True
            fz = torch.as_tensor(ores.exit_layer.reshape(B, P), dtype=torch.int32, device="cuda")
            ex, lg, nx, sim = pair.gm.prefill(tk, delta, fz)
            pair.gm.check()
            g_exit = ex.cpu().numpy()
            g_sim = sim.cpu().numpy()
        else:
            np.testing.assert_array_equal(g_exit, ores.exit_layer)
    np.testing.assert_array_equal(g_exit, ores.exit_layer)
    decisions_agree_outside_band(g_sim, ores.sim, delta, ores.exit_layer)
    out = dict(exit=g_exit, sim=g_sim, logits=lg.cpu().numpy(), next=nx.cpu().numpy(),
               final=pair.gm.final_states(B * P).cpu().numpy(), forced_rerun=forced_rerun)
    return ores, cache, out


def check_classifier_logits(pair: Pair, g_final_cls, g_logits, o_final_cls, o_logits):
    """Encoder classifier logits (a handful of outputs per sequence).

    * The head alone: the GPU's logits equal the oracle's pooler + classifier applied to the
      GPU's own final state of position 0, within the precision tolerance.
    * End to end: each row's error against the oracle, relative to the scale of the
      classifier's dot products, ||pooled|| max_c ||W_cls,c||.  With two random-init classes
      the logits are typically ~25x below that scale (their dot products cancel), so a state
      error far inside the hidden-state tolerance moves them by several times the tolerance
      relative to their own norm; the scale is the norm-wise bound of that sensitivity."""
    om = pair.om
    assert_rows_close(g_logits, om.cls_logits(np.asarray(g_final_cls, dtype=np.float64)), pair.tol,
                      "classifier logits of the GPU's own final states")
    pooled = np.tanh(om.rb(o_final_cls) @ om.w["pool.w"].T + om.w["pool.b"])
    scale = np.linalg.norm(om.rb(pooled), axis=1) * np.max(np.linalg.norm(om.w["cls.w"], axis=1))
    err = np.linalg.norm(np.asarray(g_logits, dtype=np.float64) - o_logits, axis=1) / np.maximum(scale, 1e-30)
    assert err.max() <= pair.tol, f"classifier logits: max row error {err.max():.3e} of the dot-product scale"
    return float(err.max())


def compare_prefill(pair: Pair, tokens, delta, forced=None, hsm_identity=False, check_cache=True, metric="global",
                    all_at_once=False, stop_entirely=False):
    B, P = tokens.shape
    ores, cache, g = run_prefill(pair, tokens, delta, forced, hsm_identity, metric, all_at_once, stop_entirely)
    assert_rows_close(g["final"], ores.final, pair.tol, "final states")
    if pair.cfg.family == synth.BERT:
        check_classifier_logits(pair, g["final"].reshape(B, P, -1)[:, 0], g["logits"],
                                ores.final.reshape(B, P, -1)[:, 0], ores.logits)
    else:
        assert_rows_close(g["logits"], ores.logits, pair.tol, "logits")
        check_greedy(g["next"], g["logits"], ores.logits)
    if check_cache:
        pair.compare_cache(cache, B, P)
    return ores, cache, g


def check_greedy(g_next, g_logits, o_logits):
    """The GPU's greedy token is the argmax of its own logits (lowest index on ties), and
    equals the oracle's wherever the oracle's top-2 margin exceeds twice the measured
    logit error of that row (so that no rounding difference can swap them)."""
    g = np.asarray(g_logits, dtype=np.float64)
    o = np.asarray(o_logits, dtype=np.float64)
    np.testing.assert_array_equal(np.asarray(g_next), np.argmax(g, axis=1))
    srt = np.sort(o, axis=1)
    margin = srt[:, -1] - srt[:, -2]
    sure = margin > 2 * np.max(np.abs(g - o), axis=1)
    np.testing.assert_array_equal(np.asarray(g_next)[sure], np.argmax(o, axis=1)[sure])
    return int(sure.sum())


def compare_decode(pair: Pair, cache: O.OracleCache, first_tokens, steps: int, delta: float, forced_steps=None,
                   hsm_identity=False, metric="global"):
    """Greedy decode for `steps` steps, fed with the oracle's tokens (teacher forcing), so
    both sides stay on one trajectory; per step: exit layers, similarities, final states,
    logits and greedy tokens; at the end every cached position of every layer."""
    B = len(first_tokens)
    tok = np.asarray(first_tokens)
    for s in range(steps):
        f = None if forced_steps is None else np.asarray(forced_steps[s])
        o = O.decode_step(pair.om, cache, tok, delta, f, hsm_mode="identity" if hsm_identity else "hsm", metric=metric,
                          cross=pair.cross)
        use_forced = f
        if f is None and band_tokens(o.sim, delta).any():
            use_forced = o.exit_layer
        tt = torch.as_tensor(tok, dtype=torch.int32, device="cuda")
        ft = None if use_forced is None else torch.as_tensor(use_forced, dtype=torch.int32, device="cuda")
        ex, lg, nx, sim = pair.gm.decode_step(tt, delta, ft)
        pair.gm.check()
        np.testing.assert_array_equal(ex.cpu().numpy(), o.exit_layer)
        decisions_agree_outside_band(sim.cpu().numpy(), o.sim, delta, o.exit_layer)
        assert_rows_close(pair.gm.final_states(B).cpu().numpy(), o.final, pair.tol, f"decode {s} final")
        assert_rows_close(lg.cpu().numpy(), o.logits, pair.tol, f"decode {s} logits")
        check_greedy(nx.cpu().numpy(), lg.cpu().numpy(), o.logits)
        tok = o.next_token
    return cache
