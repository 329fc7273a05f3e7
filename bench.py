#!/usr/bin/env python
"""Benchmark of the early-exit forward pass on one GB300 (N GPUs: independent replicas).

Workload (one step): a Llama-2-7B-shaped decoder in bf16 (32 layers, D=4096, 32 heads x 128,
SwiGLU 11008, vocabulary 32000, the 36 D^2 mapper, random-init N(0, 0.02)); a prompt pass over
one 2048-token prompt of uniform random ids, then 256 greedy generation steps; each token's
exit layer is forced from a normal law N(24, 4) truncated to [8, 32] (32 = full depth), paged
KV cache in 16-token blocks.  value = (prompt + generated tokens) / s over the timed steps,
inputs resident in HBM, L2 flushed between steps (every step also streams ~13 GB of weights,
far above L2).  e2e: the same steps through the C ABI with the inputs copied from pinned host
memory and the exit layers and greedy tokens copied back inside the timed region.

Also reported: the same library forced to full depth and with the identity mapper (the
speed-up the exits buy against the algorithmic ratio); the skipped-layer KV fill at Llama-7B
layer shapes on a grid of exited-token counts and exit layers, against its roofline; the
GPT-2-small workload (8 x 512-token prompts + 128 steps, exits ~ U{4..12}), threshold
calibration and the exit-rule variants on it; the BERT-base classification batch; the mapper
training steps; and the CPU oracle on a bounded sample of the Llama workload.

--impl reference times that oracle (the slow plain statement of the method) as the
reference arm.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402

PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM bytes (read + write) over algorithmic bytes of a kernel class, from one ncu capture of
# the current kernel at the workload's layer shapes (profiles/gemm_stream_llama_layer_shapes.md:
# the QKV and gate/up launches of a generation step, 104.36 + 184.19 MB of DRAM traffic for
# 100.69 + 180.39 MB of weights, rows and outputs); the line's traffic is this ratio times the
# class's algorithmic bytes per launch (traffic grows with the weight bytes streamed).
NCU_TRAFFIC_RATIO = {"gemm_decode": (104.36 + 184.19) / (100.69 + 180.39)}
METRIC = "early-exit prefill+decode tokens/s at 1 GB300; skipped-layer KV-fill % of roofline"
# Llama-7B headline workload: one prompt of LP tokens, LSTEPS greedy steps, exits ~ N(24, 4) on [8, 32]
LP, LSTEPS, LMEAN, LSD, LLO, LHI = 2048, 256, 24.0, 4.0, 8, 32
# GPT-2-small extra: B x P prompts, STEPS steps, exits ~ U{LO..HI}
B, P, STEPS, LO, HI, DELTA = 8, 512, 128, 4, 12, 0.9
L2_BYTES = 129 * 2 ** 20


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return PEAKS_FALLBACK, "fallback"


def workload_cfg():
    return synth.gpt2_small_config(max_batch=B, max_seq=P + STEPS, max_pos=1024)


# ----------------------------------------------------------------------------- algorithmic work

def gemm_work(M, N, K, esz=2, extra_out_bytes=0, extra_in_bytes=0):
    """(flops, bytes) of C[M,N] = A[M,K] B[N,K]^T: weights read once, A read, C written."""
    if M <= 0:
        return 0.0, 0.0
    return 2.0 * M * N * K, float(N * K * esz + M * K * esz + extra_out_bytes + extra_in_bytes)


def pass_work(cfg, exit_layers, decode: bool, n_seq: int = B, hsm: bool = True):
    """Algorithmic (flops, bytes) of the GEMMs of one pass given each token's exit layer.

    Counts what the method needs: layer i's projections for the tokens active at i,
    layer i's K/V of the tokens that left before i (prompt pass), the HSM of the
    exiting tokens (hsm=False: the identity mapper, no HSM work), and the head (one row per
    sequence in a prompt pass of n_seq sequences); weights are read once per launch."""
    N, D, F = cfg.n_layers, cfg.d_model, cfg.d_ffn
    dq, dkv, m1, m2 = cfg.d_q, cfg.d_kv, cfg.hsm_m1, cfg.hsm_m2
    up = 2 * F if cfg.family == synth.LLAMA else F
    e = np.asarray(exit_layers).reshape(-1)
    fl = by = 0.0
    for i in range(1, N + 1):
        act = int(np.sum(e >= i))
        ex = int(np.sum(e < i))
        for w in (gemm_work(act, dq + 2 * dkv, D, extra_out_bytes=act * (dq + 2 * dkv) * 2),
                  gemm_work(act, D, dq, extra_out_bytes=act * D * 8),
                  gemm_work(act, up, D, extra_out_bytes=act * F * 2),
                  gemm_work(act, D, F, extra_out_bytes=act * D * 8)):
            fl += w[0]
            by += w[1]
        if not decode and ex > 0 and i >= 3:
            fl += 2.0 * ex * 2 * dkv * D
            by += ex * D * 2 + ex * 2 * dkv * 2
        E = int(np.sum(e == i)) if i < N and hsm else 0
        if not decode and E > 0:
            for w in (gemm_work(E, m1, D), gemm_work(E, m2, m1), gemm_work(E, m1, m2), gemm_work(E, D, m1)):
                fl += w[0]
                by += w[1]
    if decode and hsm:
        E = int(np.sum(e < N))
        for w in (gemm_work(E, m1, D), gemm_work(E, m2, m1), gemm_work(E, m1, m2), gemm_work(E, D, m1)):
            fl += w[0]
            by += w[1]
    rows = len(e) if decode else n_seq
    w = gemm_work(rows, cfg.vocab, D, extra_out_bytes=rows * cfg.vocab * 4)
    return fl + w[0], by + w[1]


def decode_fill_work(cfg, exit_layers):
    """Grouped skipped-layer fill at the end of a generation step: (flops, bytes)."""
    N, D, dkv = cfg.n_layers, cfg.d_model, cfg.d_kv
    e = np.asarray(exit_layers).reshape(-1)
    fl = by = 0.0
    for r in range(3, N + 1):
        n = int(np.sum(e < r))
        if n:
            fl += 2.0 * n * 2 * dkv * D
            by += 2 * dkv * D * 2 + n * D * 2 + n * 2 * dkv * 2
    return fl, by


def attention_decode_work(cfg, exit_layers, keys):
    """Generation-step attention: every token active at layer i reads the K and V of its
    `keys` cached positions at that layer once.  (flops, bytes)."""
    N, dq, dkv = cfg.n_layers, cfg.d_q, cfg.d_kv
    e = np.asarray(exit_layers).reshape(-1)
    fl = by = 0.0
    for i in range(1, N + 1):
        act = int(np.sum(e >= i))
        fl += act * 4.0 * keys * dq
        by += act * (keys * 2 * dkv * 2 + 2 * dq * 2)
    return fl, by


def fill_micro_work(T, istar, n_layers=32, d=4096, dkv=4096):
    """Skipped-layer fill of T tokens exiting at i*, all deeper layers: flops and the
    algorithmic bytes (each layer's W_K/W_V once, s~ once, K/V written once)."""
    L = n_layers - istar
    flops = 2.0 * T * L * d * 2 * dkv
    bytes_ = L * 2 * dkv * d * 2 + T * d * 2 + T * L * 2 * dkv * 2
    return flops, bytes_


# ----------------------------------------------------------------------------- clocks

class Clocks:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.p = None
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        out = {"sm_mhz": None, "sm_max_mhz": None, "reasons": []}
        if self.p is None:
            out["reasons"] = ["nvidia-smi unavailable"]
            return out
        time.sleep(0.25)
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [l.strip().split(", ") for l in self.f.read().splitlines() if l.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
                for k, n in enumerate(names):
                    if r[5 + k].strip().lower() == "active":
                        reasons.add(n)
            except Exception:
                continue
        if sm:
            srt = sorted(sm)
            top = [s for s in srt if s >= 0.5 * srt[-1]] or srt
            out["sm_mhz"] = float(np.median(top))
            out["sm_max_mhz"] = max(mx)
            out["samples"] = len(sm)
        out["reasons"] = sorted(reasons)
        return out


# ----------------------------------------------------------------------------- our arm

def make_inputs(cfg, device):
    """GPT-2-small workload inputs: B x P prompt ids, prompt and generation-step exit layers."""
    tokens = synth.make_tokens(0, B, P, cfg.vocab).to(device)
    fp = synth.forced_exits_uniform(0, B * P, LO, HI, name="forced_prompt").view(B, P).to(device)
    fd = synth.forced_exits_uniform(0, STEPS * B, LO, HI, name="forced_decode").view(STEPS, B).to(device)
    return tokens, fp, fd


def llama_cfg():
    return synth.llama7b_config(max_batch=1, max_seq=LP + LSTEPS, max_pass_tokens=LP)


def llama_inputs(cfg, device):
    """Llama workload inputs: LP prompt ids, LP prompt and LSTEPS generation-step exit layers
    ~ N(LMEAN, LSD) truncated to [LLO, LHI]."""
    tok = synth.make_tokens(0, 1, LP, cfg.vocab).to(device)
    fp = synth.forced_exits_truncnorm(0, LP, LMEAN, LSD, LLO, LHI, name="forced_prompt").view(1, LP).to(device)
    fd = synth.forced_exits_truncnorm(0, LSTEPS, LMEAN, LSD, LLO, LHI, name="forced_decode").view(LSTEPS, 1).to(device)
    return tok, fp, fd


class Runner:
    """The GPT-2-small workload: B x P prompt pass, then STEPS generation steps."""

    def __init__(self, adept, cfg, device):
        self.a = adept
        self.cfg = cfg
        W = synth.make_weights(cfg, seed=0, device=device)
        self.m = adept.Model(cfg, W)
        del W
        torch.cuda.empty_cache()
        self.tokens, self.fp, self.fd = make_inputs(cfg, device)
        self.exit_p = torch.empty(B * P, dtype=torch.int32, device=device)
        self.exit_d = torch.empty(STEPS, B, dtype=torch.int32, device=device)
        self.logits = torch.empty(B, cfg.vocab, dtype=torch.float32, device=device)
        self.nxt = torch.empty(STEPS + 1, B, dtype=torch.int32, device=device)

    def step(self, delta=DELTA, threshold=False):
        a, h = self.a, self.m.h
        a.adept_prefill(h, B, P, self.tokens.view(-1), delta, None if threshold else self.fp.view(-1), self.exit_p,
                        self.logits, self.nxt[0], None)
        for s in range(STEPS):
            a.adept_decode_step(h, B, self.nxt[s], delta, None if threshold else self.fd[s], self.exit_d[s],
                                self.logits, self.nxt[s + 1], None)


class LlamaRunner:
    """The headline step at the Llama-2-7B shape: one LP-token prompt pass and LSTEPS greedy
    generation steps through the C ABI."""

    def __init__(self, adept, device):
        self.a = adept
        self.cfg = cfg = llama_cfg()
        W = synth.make_weights(cfg, seed=0, device=device)
        self.m = adept.Model(cfg, W)
        del W
        torch.cuda.empty_cache()
        self.tok, self.fp, self.fd = llama_inputs(cfg, device)
        self.exit_p = torch.empty(LP, dtype=torch.int32, device=device)
        self.exit_d = torch.empty(LSTEPS, 1, dtype=torch.int32, device=device)
        self.nxt = torch.empty(LSTEPS + 1, 1, dtype=torch.int32, device=device)

    def prefill(self, tok=None, fp=None):
        self.a.adept_prefill(self.m.h, 1, LP, (self.tok if tok is None else tok).view(-1), DELTA,
                             (self.fp if fp is None else fp).view(-1), self.exit_p, None, self.nxt[0], None)

    def decode(self, fd=None):
        fd = self.fd if fd is None else fd
        for s in range(LSTEPS):
            self.a.adept_decode_step(self.m.h, 1, self.nxt[s], DELTA, fd[s], self.exit_d[s], None, self.nxt[s + 1],
                                     None)

    def step(self, tok=None, fp=None, fd=None):
        self.prefill(tok, fp)
        self.decode(fd)


def run_fill_micro(adept, device, peaks, grid_T, grid_i, reps=3):
    """Skipped-layer fill through adept_skip_kv_fill at Llama-7B layer shapes."""
    Tmax = max(grid_T)
    seqs = 32
    cfg = synth.llama7b_config(max_batch=seqs, max_seq=max(2048, (Tmax + seqs - 1) // seqs), max_pass_tokens=64,
                               block_shuffle_seed=1234)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    torch.cuda.empty_cache()
    adept.adept_seq_reserve(m.h, [cfg.max_seq] * seqs)
    h_all = synth.make_mapped_states(5, Tmax, cfg.d_model, device=device)
    j = torch.arange(Tmax, device=device, dtype=torch.int32)
    seq_all = (j % seqs).to(torch.int32).contiguous()
    pos_all = (j // seqs).to(torch.int32).contiguous()
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
    rows = []
    st = torch.cuda.current_stream()
    # cells in increasing work (T ascending; within a T, fewer layers to fill first), so that no
    # short cell follows a long, power-heavy one (the T = 65536 cells run 25-90 ms tensor-bound)
    for T in sorted(grid_T):
        for istar in sorted(grid_i, reverse=True):
            el = torch.full((T,), istar, dtype=torch.int32, device=device)
            args = (m.h, T, h_all[:T].contiguous(), el, seq_all[:T].contiguous(), pos_all[:T].contiguous())
            adept.adept_skip_kv_fill(*args)
            torch.cuda.synchronize()
            # the call as a user makes it (programmatic dependent launch, no per-launch events),
            # enqueued back to back so that the host's preparation of a call overlaps the device
            # work before it (the L2 flush): the events time the device's work for the call
            evs = []
            for _ in range(reps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(st)
                adept.adept_skip_kv_fill(*args)
                e1.record(st)
                evs.append((e0, e1))
            torch.cuda.synchronize()
            ts = [a.elapsed_time(b) for a, b in evs]
            # the GEMM launch alone, event-bracketed in a profiled call (informational)
            adept.adept_set_option(m.h, adept.OPT_PROFILE, 1)
            adept.adept_profile_read(m.h, adept.PROF_KV_FILL)
            for _ in range(reps):
                flush.zero_()
                adept.adept_skip_kv_fill(*args)
                torch.cuda.synchronize()
            n, kms, _, _ = adept.adept_profile_read(m.h, adept.PROF_KV_FILL)
            adept.adept_set_option(m.h, adept.OPT_PROFILE, 0)
            adept.adept_check_device_status(m.h)
            fl, by = fill_micro_work(T, istar)
            t = float(np.median(ts)) / 1e3
            tk = kms / max(n, 1) / 1e3
            t_f, t_b = fl / (peaks["bf16_tflops"] * 1e12), by / (peaks["hbm_gbs"] * 1e9)
            roof = max(t_f, t_b)
            row = {"T": T, "exit_layer": istar, "ms": round(t * 1e3, 4), "gemm_ms": round(tk * 1e3, 4),
                   "tflops": round(fl / t / 1e12, 2), "gbs": round(by / t / 1e9, 1),
                   "roofline_ms": round(roof * 1e3, 4), "frac": round(roof / t, 4),
                   "bound": "tensor" if t_f > t_b else "hbm"}
            if t_f > t_b:   # a long tensor-bound launch also against the sustained bf16 peak
                roof_s = max(fl / (peaks["bf16_tflops_sustained"] * 1e12), t_b)
                row["frac_of_sustained"] = round(roof_s / t, 4)
            rows.append(row)
    m.close()
    rows.sort(key=lambda r: (r["exit_layer"], r["T"]))
    del h_all
    torch.cuda.empty_cache()
    return rows


def llama_work(cfg, exit_prompt, exit_decode, hsm: bool = True):
    """Algorithmic flops of a one-sequence Llama-shaped prompt pass + generation steps (GEMMs,
    fills, HSM unless hsm=False, head) from the exit layers: the cost the early exit saves or
    adds."""
    fl = pass_work(cfg, exit_prompt, decode=False, n_seq=1, hsm=hsm)[0]
    for e in exit_decode:
        fl += pass_work(cfg, e, decode=True, hsm=hsm)[0] + decode_fill_work(cfg, e)[0]
    return fl


def run_encoder(adept, device, B=64, P=128):
    """BERT-base shape, bf16, random-init: 64 x 128-token classification batch.  Threshold
    exits at delta = 0.9 (the configuration's threshold; with random-init weights every token
    leaves at the first eligible layer there), at the delta that threshold calibration finds
    for a 25 % reduction in computation on this batch, forced exits ~ U{4..12}, and full depth;
    the default exit (deeper K/V filled from s~) against the encoder's "stop entirely" variant
    (Sec. 4.3).  Throughput in sequences/s and tokens/s including the classifier."""
    cfg = synth.bert_base_config(max_batch=B, max_seq=P, max_pass_tokens=B * P)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    tok = synth.make_tokens(0, B, P, cfg.vocab).to(device)
    fz = synth.forced_exits_uniform(0, B * P, 4, 12, name="forced_encoder").view(-1).to(device)
    full = torch.full_like(fz, cfg.n_layers)
    ex = torch.empty(B * P, dtype=torch.int32, device=device)
    lg = torch.empty(B, cfg.n_classes, device=device)
    st = torch.cuda.current_stream()
    d_c, r_c, n_c = adept.adept_calibrate_threshold(m.h, B, P, tok.view(-1), 0.25, 0.01, 24)
    out = {}
    for name, forced, stop, delta in (("threshold_0.9", None, 0, 0.9), ("threshold_calibrated", None, 0, d_c),
                                      ("forced_U4_12", fz, 0, 0.9), ("forced_U4_12_stop_entirely", fz, 1, 0.9),
                                      ("full_depth", full, 0, 0.9)):
        adept.adept_set_option(m.h, adept.OPT_STOP_ENTIRELY, stop)
        ts = []
        for rep in range(4):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(st)
            adept.adept_prefill(m.h, B, P, tok.view(-1), delta, forced, ex, lg, None, None)
            e1.record(st)
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        t = float(np.median(ts[1:])) / 1e3
        out[name] = {"ms": round(t * 1e3, 3), "seq_s": round(B / t, 1), "tok_s": round(B * P / t, 1),
                     "mean_exit_depth": round(float(ex.double().mean().item()), 3)}
        if name == "threshold_calibrated":
            out[name].update(delta=round(d_c, 6), rdc=round(r_c, 4), calibration_passes=n_c)
    adept.adept_set_option(m.h, adept.OPT_STOP_ENTIRELY, 0)
    adept.adept_check_device_status(m.h)
    m.close()
    torch.cuda.empty_cache()
    return {"workload": f"BERT-base shape, bf16, random-init; {B} x {P}-token classification batch", **out}


def run_encdec(adept, device, B=8, S=256, T=8, steps=8, reps=4):
    """OFA-base-shaped encoder-decoder (Sec. 5.2; 6 + 6 layers, D 768, 12 heads, FFN 3072,
    bf16, random-init): B sequences of S source tokens (a text stand-in for OFA's image and
    text source), a T-token target prompt and `steps` greedy steps.  One pass = the encoder's
    prompt pass, the decoder's source K/V (adept_set_cross_source from the encoder's final
    states, on the device), the decoder's prompt pass and its generation steps.  Exits ~ U{2..6}
    per token in both stacks against full depth; tokens/s counts source + target tokens."""
    enc, dec = synth.ofa_base_configs(src_len=S, tgt_len=T + steps, batch=B)
    me = adept.Model(enc, synth.make_weights(enc, seed=0, device=device))
    md = adept.Model(dec, synth.make_weights(dec, seed=1, device=device))
    src = synth.make_tokens(0, B, S, enc.vocab).to(device)
    tgt = synth.make_tokens(1, B, T, dec.vocab).to(device)
    fe = synth.forced_exits_uniform(0, B * S, 2, enc.n_layers, name="forced_enc").view(B, S).to(device)
    fd = synth.forced_exits_uniform(1, B * T, 2, dec.n_layers, name="forced_dec").view(B, T).to(device)
    fs = synth.forced_exits_uniform(2, B * steps, 2, dec.n_layers, name="forced_steps").view(steps, B).to(device)
    st = torch.cuda.current_stream()
    fin = torch.empty(B * S, enc.d_model, device=device)

    def one(full):
        ex_e, _, _, _ = me.prefill(src, 0.9, torch.full_like(fe, enc.n_layers) if full else fe)
        adept.adept_read_final_states(me.h, fin, B * S)
        md.set_cross_source([S] * B, fin)
        ex_d, _, nx, _ = md.prefill(tgt, 0.9, torch.full_like(fd, dec.n_layers) if full else fd)
        for k in range(steps):
            f = torch.full_like(fs[k], dec.n_layers) if full else fs[k]
            _, _, nx, _ = md.decode_step(nx.view(-1).contiguous(), 0.9, f.contiguous())
        return ex_e, ex_d

    out = {}
    for name, full in (("early_exit", False), ("full_depth", True)):
        ts = []
        for _ in range(reps):
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            ex_e, ex_d = one(full)
            e1.record(st)
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        t = float(np.median(ts[1:])) / 1e3
        out[name] = {"ms": round(t * 1e3, 3), "tok_s": round(B * (S + T + steps) / t, 1),
                     "encoder_mean_exit": round(float(ex_e.double().mean().item()), 3),
                     "decoder_prompt_mean_exit": round(float(ex_d.double().mean().item()), 3)}
    out["speedup"] = round(out["full_depth"]["ms"] / out["early_exit"]["ms"], 4)
    me.check()
    md.check()
    me.close()
    md.close()
    torch.cuda.empty_cache()
    return {"workload": f"OFA-base-shaped encoder-decoder (6 + 6 layers, D 768), bf16, random-init; {B} x {S} source "
                        f"tokens, {T}-token target prompt + {steps} greedy steps; forced exits U{{2..6}} in both stacks",
            **out}


def hsm_train_flops(cfg, n, n_cls=0):
    """GEMM FLOPs of one HSM training step on n examples: the four FC products forward, their
    input and weight gradients (3 x 2 x FC weights per example), then for decoders the head
    forward and its input gradient (2 x 2 D V per example), for encoders the pooler forward
    and its input gradient on the n_cls labelled rows (2 x 2 D^2 per row)."""
    D, m1, m2 = cfg.d_model, cfg.hsm_m1, cfg.hsm_m2
    fc = D * m1 + m1 * m2 + m2 * m1 + m1 * D
    if cfg.family == synth.BERT:
        return n * 6.0 * fc + n_cls * 4.0 * D * D
    return n * (6.0 * fc + 4.0 * D * cfg.vocab)


def run_hsm_train(adept, device, peaks, n=8192, reps=5, shape="gpt2"):
    """HSM training step (Sec. 4.2; App. D), n synthetic examples per step, bf16 GEMM operands,
    fp32 master weights and AdamW state.  shape "gpt2": GPT-2-small (D 768, HSM widths 3072 /
    6144, vocabulary 50257; 8192 examples = 128 sequences x 64 tokens); "llama7b": Llama-2-7B
    (D 4096, HSM widths 8192 / 32768, vocabulary 32000; 8192 examples = 8 sequences x 1024
    tokens); "bert": BERT-base encoder (D 768, HSM widths 3072 / 6144, two classes; 8192
    examples = 64 sequences x 128 tokens, the 64 [CLS] rows labelled) with the similarity +
    classification loss of Sec. 4.3.  Only the frozen head and the HSM take part, so the models
    carry 2 layers.  Step time with CUDA events; the GEMMs' TFLOP/s from per-GEMM events in a
    separate profiled step."""
    n_cls = 0
    if shape == "bert":
        cfg = synth.bert_base_config(n_layers=2, max_batch=1, max_seq=16)
        desc = "BERT-base shape HSM (768 -> 3072 -> 6144 -> 3072 -> 768) + frozen pooler / 2-class classifier"
        n_cls = n // 128
    elif shape == "llama7b":
        cfg = synth.llama7b_config(n_layers=2, max_batch=1, max_seq=16)
        desc = "Llama-2-7B shape HSM (4096 -> 8192 -> 32768 -> 8192 -> 4096) + frozen 32000-token head"
    else:
        cfg = synth.gpt2_small_config(n_layers=2, max_batch=1, max_seq=16)
        desc = "GPT-2-small shape HSM (768 -> 3072 -> 6144 -> 3072 -> 768) + frozen 50257-token head"
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    adept.adept_hsm_train_init(m.h, n)
    loss = torch.zeros(1, device=device)
    st = torch.cuda.current_stream()
    if shape == "bert":
        s_i, s_prev, inertia, s_fin, lab = [x.to(device) for x in synth.hsm_cls_batch(cfg, n, n_cls, seed=1)]
        step = lambda: adept.adept_hsm_train_step_cls(m.h, n, s_i, s_prev, inertia, s_fin, lab, 1e-4,  # noqa
                                                      loss_out=loss)
    else:
        s_i, s_prev, inertia, tgt = [x.to(device) for x in synth.hsm_train_batch(cfg, n, seed=1)]
        step = lambda: adept.adept_hsm_train_step(m.h, n, s_i, s_prev, inertia, tgt, 1e-4, 0.9, 0.999, 1e-8,  # noqa
                                                  0.0, loss_out=loss)
    step()
    adept.adept_check_device_status(m.h)
    first_loss = float(loss.item())
    adept.adept_launch_count(m.h)
    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(st)
        step()
        e1.record(st)
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    launches = adept.adept_launch_count(m.h) // reps
    t = float(np.median(ts)) / 1e3
    fl = hsm_train_flops(cfg, n, n_cls)
    adept.adept_set_option(m.h, adept.OPT_PROFILE, 1)
    step()
    ng, gms, _, _ = adept.adept_profile_read(m.h, adept.PROF_GEMM_TRAIN)
    adept.adept_set_option(m.h, adept.OPT_PROFILE, 0)
    adept.adept_check_device_status(m.h)
    last_loss = float(loss.item())
    m.close()
    torch.cuda.empty_cache()
    peak = peaks["bf16_tflops_sustained"]
    return {"workload": f"{desc}, {n} examples/step, bf16 GEMM operands, fp32 AdamW",
            "ms_per_step": round(t * 1e3, 3), "examples_s": round(n / t, 1), "gpu_launches": int(launches),
            "gemm_tflop_per_step": round(fl / 1e12, 4), "tflops_step": round(fl / t / 1e12, 1),
            "gemm_launches": int(ng), "gemm_ms_profiled": round(gms, 3),
            "gemm_tflops_profiled": round(fl / (gms / 1e3) / 1e12, 1) if gms > 0 else None,
            "gemm_frac_of_measured_sustained_bf16": round(fl / (gms / 1e3) / 1e12 / peak, 4) if gms > 0 else None,
            "loss_first": round(first_loss, 5), "loss_after": round(last_loss, 5)}


def timed_prefill_decode(run, st, tok=None, fp=None, fd=None, reps=2):
    """(prompt-pass ms, generation ms per step) of the last of `reps` runs of the Llama step
    (the first warms up and captures the generation-step graph)."""
    for _ in range(reps):
        e0, e1, e2 = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        torch.cuda.synchronize()
        e0.record(st)
        run.prefill(tok, fp)
        e1.record(st)
        run.decode(fd)
        e2.record(st)
        torch.cuda.synchronize()
    return e0.elapsed_time(e1), e1.elapsed_time(e2) / LSTEPS


def llama_arms(adept, run, st):
    """The headline model against itself forced to full depth, and with the identity mapper in
    place of the HSM (s~ = s_i*: the speed-up the exits and fills alone allow)."""
    cfg = run.cfg
    full_p = torch.full_like(run.fp, cfg.n_layers)
    full_d = torch.full_like(run.fd, cfg.n_layers)
    out = {}
    for name, fp, fd in (("early_exit", run.fp, run.fd), ("full_depth", full_p, full_d), ("hsm_identity", run.fp, run.fd)):
        adept.adept_set_option(run.m.h, adept.OPT_HSM_IDENTITY, int(name == "hsm_identity"))
        tp, td = timed_prefill_decode(run, st, None, fp, fd)
        adept.adept_check_device_status(run.m.h)
        ep, ed = run.exit_p.cpu().numpy(), run.exit_d.cpu().numpy()
        out[name] = {"prefill_tok_s": round(LP / tp * 1e3, 1), "decode_tok_s": round(1e3 / td, 2),
                     "tok_s": round((LP + LSTEPS) / (tp + td * LSTEPS) * 1e3, 2), "prefill_ms": round(tp, 3),
                     "decode_ms_per_step": round(td, 4),
                     "mean_exit_depth": round(float(np.concatenate([ep, ed.reshape(-1)]).mean()), 3),
                     "algorithmic_tflop": round(llama_work(cfg, ep, ed, hsm=name != "hsm_identity") / 1e12, 3)}
    adept.adept_set_option(run.m.h, adept.OPT_HSM_IDENTITY, 0)
    ee, fd_, hi = out["early_exit"], out["full_depth"], out["hsm_identity"]
    return {"workload": "the headline workload vs all tokens forced to layer 32, and the same exits with the "
                        "identity mapper",
            **out,
            "speedup": round(ee["tok_s"] / fd_["tok_s"], 4),
            "prefill_speedup": round(fd_["prefill_ms"] / ee["prefill_ms"], 4),
            "decode_speedup": round(fd_["decode_ms_per_step"] / ee["decode_ms_per_step"], 4),
            "algorithmic_ratio": round(fd_["algorithmic_tflop"] / ee["algorithmic_tflop"], 4),
            "depth_ratio": round(fd_["mean_exit_depth"] / ee["mean_exit_depth"], 4),
            "speedup_hsm_identity": round(hi["tok_s"] / fd_["tok_s"], 4),
            "algorithmic_ratio_hsm_identity": round(fd_["algorithmic_tflop"] / hi["algorithmic_tflop"], 4)}


def run_gpt2(adept, device, reps=3):
    """GPT-2-small workload (B x P prompts + STEPS greedy steps) with forced exits ~ U{4..12}
    and in threshold mode at delta 0.9, then threshold calibration to a 25 % reduction in
    computation and the exit-rule variants at the calibrated delta (prompt passes)."""
    cfg = workload_cfg()
    run = Runner(adept, cfg, device)
    st = torch.cuda.current_stream()
    out = {"workload": "gpt2-small-shaped decoder, bf16, random-init N(0,0.02); batch 8 x 512-token uniform random "
                       "prompts + 128 greedy decode steps"}
    for name, thr in (("forced_U4_12", False), ("threshold_0.9", True)):
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(st)
            run.step(DELTA, thr)
            e1.record(st)
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        adept.adept_check_device_status(run.m.h)
        t = float(np.median(ts[1:])) / 1e3
        out[name] = {"ms_per_step": round(t * 1e3, 3), "tok_s": round((B * P + B * STEPS) / t, 1),
                     "prompt_mean_exit": round(float(run.exit_p.double().mean().item()), 3),
                     "decode_mean_exit": round(float(run.exit_d.double().mean().item()), 3)}
    # threshold calibration (Sec. 4.1, 5.1): bisection on delta to a 25 % reduction in computation
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    d_c, r_c, n_c = adept.adept_calibrate_threshold(run.m.h, B, P, run.tokens.view(-1), 0.25, 0.01, 24)
    t_cal = (time.perf_counter() - t0) * 1e3
    out["calibration"] = {"target_rdc": 0.25, "tol": 0.01, "delta": round(d_c, 6), "rdc": round(r_c, 4),
                          "passes": n_c, "ms": round(t_cal, 3), "ms_per_pass": round(t_cal / max(n_c, 1), 3),
                          "batch": f"{B} x {P} workload prompts, threshold exits"}
    # exit-rule variants (App. H.2-H.3) at the calibrated threshold
    variants = {}
    ex_v = torch.empty(B * P, dtype=torch.int32, device=device)
    nx_v = torch.empty(B, dtype=torch.int32, device=device)
    for name, metric, aao in (("global", 0, 0), ("local", 1, 0), ("both", 2, 0), ("all_at_once", 0, 1)):
        adept.adept_set_option(run.m.h, adept.OPT_EXIT_METRIC, metric)
        adept.adept_set_option(run.m.h, adept.OPT_ALL_AT_ONCE, aao)
        adept.adept_prefill(run.m.h, B, P, run.tokens.view(-1), d_c, None, ex_v, None, nx_v, None)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        adept.adept_prefill(run.m.h, B, P, run.tokens.view(-1), d_c, None, ex_v, None, nx_v, None)
        e1.record(st)
        torch.cuda.synchronize()
        depth = ex_v.double().mean().item()
        variants[name] = {"rdc": round(1.0 - depth / cfg.n_layers, 4), "prompt_ms": round(e0.elapsed_time(e1), 3)}
    adept.adept_set_option(run.m.h, adept.OPT_EXIT_METRIC, 0)
    adept.adept_set_option(run.m.h, adept.OPT_ALL_AT_ONCE, 0)
    adept.adept_check_device_status(run.m.h)
    out["exit_variants"] = {"delta": round(d_c, 6), "batch": f"{B} x {P} workload prompts", **variants}
    run.m.close()
    del run
    torch.cuda.empty_cache()
    return out


def max_over_ranks(x: float, world: int, device) -> float:
    """The slowest rank's value (replicas: the job ends when the last rank does)."""
    if world <= 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank_step: float, steps: int, world: int, seconds: float) -> float:
    """Whole-job throughput of `world` independent replicas: every rank's units over the
    slowest rank's time."""
    return world * units_per_rank_step * steps / seconds


def class_work(cfg, e_p, e_d):
    """Algorithmic (flops, bytes) of one headline step per kernel class: the prompt pass's
    GEMMs (one sequence), the generation steps' GEMMs (layers on the active token, mapper,
    head) and their grouped skipped-layer fills."""
    wd = [pass_work(cfg, e_d[s], decode=True) for s in range(len(e_d))]
    wf = [decode_fill_work(cfg, e_d[s]) for s in range(len(e_d))]
    return {"gemm_prefill": pass_work(cfg, e_p, decode=False, n_seq=1),
            "gemm_decode": (sum(w[0] for w in wd), sum(w[1] for w in wd)),
            "kv_fill_decode": (sum(w[0] for w in wf), sum(w[1] for w in wf))}


def ours(args, rank, world, device):
    import paper_2601_03700_gb300 as adept
    if not os.path.exists(adept.LIB_PATH):
        from paper_2601_03700_gb300 import build as _b
        _b.build()
    adept.load_library()
    peaks, peaks_src = load_peaks()
    run = LlamaRunner(adept, device)
    cfg = run.cfg
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=device)
    st = torch.cuda.current_stream()
    for _ in range(args.warmup):
        run.step()
    torch.cuda.synchronize()
    adept.adept_check_device_status(run.m.h)
    # --------------------------------------------------------------- timed region
    adept.adept_launch_count(run.m.h)
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    total_ms = 0.0
    for _ in range(args.steps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        run.step()
        e1.record(st)
        torch.cuda.synchronize()
        total_ms += e0.elapsed_time(e1)
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop() if clocks else None
    launches = adept.adept_launch_count(run.m.h)
    adept.adept_check_device_status(run.m.h)
    total_ms = max_over_ranks(total_ms, world, device)
    tok_per_step = LP + LSTEPS
    value = replica_throughput(tok_per_step, args.steps, world, total_ms / 1e3)
    ms_per_step = total_ms / args.steps
    # --------------------------------------------------------------- end-to-end through the API with host buffers
    tok_h, fp_h, fd_h = run.tok.cpu().pin_memory(), run.fp.cpu().pin_memory(), run.fd.cpu().pin_memory()
    nxt_h = torch.empty(LSTEPS + 1, 1, dtype=torch.int32).pin_memory()
    ex_h = torch.empty(LP + LSTEPS, dtype=torch.int32).pin_memory()
    tok_d, fp_d, fd_d = torch.empty_like(run.tok), torch.empty_like(run.fp), torch.empty_like(run.fd)
    e2e_t = 0.0
    n_e2e = max(1, args.steps)
    for _ in range(n_e2e):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        tok_d.copy_(tok_h, non_blocking=True)
        fp_d.copy_(fp_h, non_blocking=True)
        fd_d.copy_(fd_h, non_blocking=True)
        run.step(tok_d, fp_d, fd_d)
        nxt_h.copy_(run.nxt, non_blocking=True)
        ex_h[:LP].copy_(run.exit_p, non_blocking=True)
        ex_h[LP:].copy_(run.exit_d.view(-1), non_blocking=True)
        torch.cuda.synchronize()
        e2e_t += time.perf_counter() - t0
    e2e_t = max_over_ranks(e2e_t, world, device)
    e2e = replica_throughput(tok_per_step, n_e2e, world, e2e_t)
    h2d = (tok_h.numel() + fp_h.numel() + fd_h.numel()) * 4
    d2h = (nxt_h.numel() + ex_h.numel()) * 4
    # --------------------------------------------------------------- one step with the span timer (in-situ kernel time)
    # The weight-streaming GEMM launches (the generation steps' layer, mapper and head GEMMs, and
    # their grouped skipped-layer fills) record their spans on the device timer while the step
    # runs as timed (programmatic dependent launch, graph replay): from the first CTA past the
    # grid-dependency wait to the end of the last thread.  Consecutive launches' spans do not
    # overlap, so a class's summed span never exceeds the step.
    adept.adept_set_option(run.m.h, adept.OPT_SPAN_TIMER, 1)
    run.step()   # graphs are captured again with the span sites
    torch.cuda.synchronize()
    for c in range(adept.PROF_GEMM_TRAIN + 1):
        adept.adept_span_read(run.m.h, c)
    flush.zero_()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    run.step()
    e1.record(st)
    torch.cuda.synchronize()
    span_step_ms = e0.elapsed_time(e1)
    spans = {c: adept.adept_span_read(run.m.h, c) for c in range(adept.PROF_GEMM_TRAIN + 1)}
    adept.adept_set_option(run.m.h, adept.OPT_SPAN_TIMER, 0)
    adept.adept_check_device_status(run.m.h)
    # --------------------------------------------------------------- dominant kernel roofline
    e_p = run.exit_p.cpu().numpy()
    e_d = run.exit_d.cpu().numpy()
    work = class_work(cfg, e_p, e_d)
    names = {adept.PROF_GEMM_DECODE: "gemm_decode", adept.PROF_KV_FILL: "kv_fill_decode"}
    per_class = {names[c]: {"launches": spans[c][0], "span_ms_per_step": round(spans[c][1], 4),
                            "share_of_step": round(spans[c][1] / span_step_ms, 4)} for c in names}
    dom_c = max(names, key=lambda c: spans[c][1])
    dom = names[dom_c]
    n, ms = spans[dom_c]
    fl, by = work[dom]
    t_f = fl / (peaks["bf16_tflops"] * 1e12)
    t_b = by / (peaks["hbm_gbs"] * 1e9)
    if t_f >= t_b:
        roof = {"bound": "tensor", "achieved": round(fl / (ms / 1e3) / 1e12, 3), "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s"}
    else:
        roof = {"bound": "hbm", "achieved": round(by / (ms / 1e3) / 1e9, 2), "peak": peaks["hbm_gbs"], "unit": "GB/s"}
    roof["frac"] = round(roof["achieved"] / roof["peak"], 4)
    tr = NCU_TRAFFIC_RATIO.get(dom)
    roof["traffic"] = round(tr * by / max(n, 1)) if tr else None
    roof["traffic_source"] = "ncu DRAM bytes / algorithmic bytes of the captured launches x algorithmic bytes per launch"
    roof["kernel"] = dom + " (stream-K and cluster K-split weight-streaming GEMM launches)"
    roof["launches"] = n
    roof["peak_source"] = (peaks_src + " (MEASURED_PEAKS.json)") if peaks_src == "measured" else peaks_src
    roof["timing"] = ("device-timer span per launch (first CTA past the grid-dependency wait to the last thread's "
                      "end), summed over the class in one step run as timed (PDL, graph replay) after the timed steps")
    roof["class_ms_per_step"] = round(ms, 3)
    roof["class_share_of_step"] = round(ms / span_step_ms, 4)
    roof["span_step_ms"] = round(span_step_ms, 3)
    roof["work_per_launch"] = {"flop": round(fl / max(n, 1)), "bytes": round(by / max(n, 1))}
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "Llama-2-7B-shaped decoder, bf16, random-init N(0,0.02); batch 1, 2048-token uniform "
                               "random prompt + 256 greedy decode steps; forced exit layer per token ~ N(24,4) "
                               "truncated to [8,32]; paged KV cache, 16-token blocks",
                   "model": "llama2-7b-shape", "global_batch": world, "seq_len": LP, "decode_steps": LSTEPS,
                   "parallelism": f"replicas{world}" if world > 1 else "single",
                   "l2": "flushed between timed steps (256 MiB write); each step streams ~13 GB of weights"},
        "e2e": {"value": round(e2e, 2), "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "roofline": roof,
        "kernel_classes": per_class,
        "exit_depth": {"prompt_mean": round(float(e_p.mean()), 3), "decode_mean": round(float(e_d.mean()), 3)},
        "clocks": clk,
    }
    if rank == 0 and not args.no_llama:
        line["llama7b_arms"] = llama_arms(adept, run, st)
    run.m.close()
    del run
    torch.cuda.empty_cache()
    if rank == 0 and not args.no_kv_fill:
        grid_T = [int(x) for x in args.fill_T.split(",")]
        grid_i = [int(x) for x in args.fill_i.split(",")]
        rows = run_fill_micro(adept, device, peaks, grid_T, grid_i)
        fr = [r["frac"] for r in rows]
        line["kv_fill"] = {"shape": "Llama-7B layers: 32 x (D=4096 -> K,V 2x4096), bf16, paged 16-token blocks",
                           "peak": {"tflops": peaks["bf16_tflops"], "tflops_sustained": peaks["bf16_tflops_sustained"],
                                    "gbs": peaks["hbm_gbs"], "source": peaks_src},
                           "mean_frac": round(float(np.mean(fr)), 4), "min_frac": round(float(np.min(fr)), 4),
                           "cells_below_0.6": int(sum(f < 0.6 for f in fr)), "grid": rows}
        line["kv_fill_frac"] = {"mean": line["kv_fill"]["mean_frac"], "min": line["kv_fill"]["min_frac"],
                                "cells": len(rows)}
    if rank == 0 and not args.no_llama:
        line["gpt2_small"] = run_gpt2(adept, device)
        line["encoder"] = run_encoder(adept, device)
        line["encoder_decoder"] = run_encdec(adept, device)
        line["hsm_train"] = run_hsm_train(adept, device, peaks)
        line["hsm_train_llama7b"] = run_hsm_train(adept, device, peaks, shape="llama7b", reps=3)
        line["hsm_train_bert"] = run_hsm_train(adept, device, peaks, shape="bert")
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.cpu_tokens, args.cpu_steps)
    return line


# ----------------------------------------------------------------------------- oracle (CPU) arms

def host_mem_available() -> int:
    """MemAvailable of the host in bytes (0 when unknown)."""
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith("MemAvailable:"):
                    return int(ln.split()[1]) * 1024
    except Exception:
        pass
    return 0


# fp64 oracle copy of the Llama-7B-shaped model: 7.3e9 weights x 8 B
ORACLE_LLAMA_BYTES = 59 * 2 ** 30


class _WeightStream:
    """The workload's weights as a mapping whose items() generates one tensor at a time (on
    the GPU when there is one: the same values bit for bit), so the oracle's fp64 copy is the
    only full copy of the model in host memory."""

    def __init__(self, cfg):
        self.cfg = cfg
        self.dev = "cuda" if torch.cuda.is_available() else "cpu"

    def items(self):
        for name, shape in synth.weight_shapes(self.cfg).items():
            yield name, synth.make_weight(self.cfg, name, shape, seed=0, device=self.dev).cpu()


def oracle_llama_model():
    """(cfg, oracle model) of the headline workload."""
    from oracle import adept_oracle as O
    cfg = llama_cfg()
    om = O.OracleModel(cfg, _WeightStream(cfg))
    if torch.cuda.is_available():
        torch.cuda.empty_cache()
    return cfg, om


def oracle_sample(n_seq: int, prompt: int, steps: int, model=None):
    """Runs the oracle on a bounded sample of a workload: n_seq prompts of `prompt` tokens and
    `steps` generation steps, same model, same exit law.  model = (cfg, oracle model) of the
    Llama workload (prompt ids and exit layers are the workload's leading ones); None: the
    GPT-2-small workload.  Returns (tokens processed, seconds)."""
    from oracle import adept_oracle as O
    if model is None:
        cfg = workload_cfg()
        W = synth.make_weights(cfg, seed=0)
        om = O.OracleModel(cfg, W)
        del W
        tokens, fp, fd = make_inputs(cfg, "cpu")
    else:
        cfg, om = model
        tokens, fp, fd = llama_inputs(cfg, "cpu")
    tk = tokens[:n_seq, :prompt].numpy()
    f = fp[:n_seq, :prompt].numpy()
    cache = O.OracleCache(cfg, n_seq, prompt + steps + 1)
    t0 = time.perf_counter()
    r = O.prefill(om, cache, tk, DELTA, f)
    nxt = r.next_token
    for s in range(steps):
        r = O.decode_step(om, cache, nxt, DELTA, fd[s, :n_seq].numpy())
        nxt = r.next_token
    dt = time.perf_counter() - t0
    return n_seq * (prompt + steps), dt


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def llama_oracle_fits() -> bool:
    return host_mem_available() >= 1.4 * ORACLE_LLAMA_BYTES


def cpu_baseline(prompt: int, steps: int):
    """The oracle on the host cores, on a bounded sample of the headline workload (the Llama
    model with the workload's first `prompt` prompt tokens and `steps` generation steps).  Where
    the host cannot hold the oracle's fp64 copy of that model, the GPT-2-small workload stands in
    (said in `sample`)."""
    if llama_oracle_fits():
        t0 = time.perf_counter()
        model = oracle_llama_model()
        t_build = time.perf_counter() - t0
        tok, dt = oracle_sample(1, prompt, steps, model)
        out = {"value": round(tok / dt, 3), "unit": "tokens/s", "cores": cores(), "kind": "oracle",
               "sample": f"Llama-2-7B-shaped model of the workload, its first {prompt} prompt tokens + {steps} "
                         f"generation steps, same exit law (fp64 NumPy oracle, {dt:.1f} s; model build "
                         f"{t_build:.0f} s untimed)"}
        del model
    else:
        tok, dt = oracle_sample(4, 512, 8)
        out = {"value": round(tok / dt, 3), "unit": "tokens/s", "cores": cores(), "kind": "oracle",
               "sample": f"host memory below the fp64 Llama-7B oracle's ~75 GB: GPT-2-small workload instead, "
                         f"4 prompts x 512 tokens + 8 generation steps ({dt:.1f} s)"}
    out["single_core"] = oracle_single_core(1, 128, 8)
    return out


def oracle_single_core(n_seq: int, prompt: int, steps: int):
    """The oracle on one host core (GPT-2-small workload): a fresh interpreter with every BLAS /
    OpenMP pool limited to one thread, on a smaller bounded sample."""
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
        env[k] = "1"
    env["CUDA_VISIBLE_DEVICES"] = ""
    try:
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample", f"{n_seq},{prompt},{steps}"],
                           env=env, capture_output=True, text=True, timeout=600)
        d = json.loads([x for x in r.stdout.splitlines() if x.startswith("{")][-1])
    except Exception as e:   # reported, not fatal: the all-core figure stands
        return {"unavailable": f"{type(e).__name__}: {e}"[:200]}
    return {"value": round(d["tokens"] / d["seconds"], 3), "unit": "tokens/s", "cores": 1,
            "sample": f"GPT-2-small workload, {n_seq} prompt x {prompt} tokens + {steps} decode steps "
                      f"({d['seconds']:.1f} s)"}


def reference_arm(args, rank, world):
    """The oracle as the reference arm: each step a bounded sample of the headline workload
    (its first --ref-prompt prompt tokens and --ref-steps generation steps on the Llama model;
    the GPT-2-small workload where the host cannot hold the fp64 Llama model)."""
    if rank != 0:
        return None
    llama = llama_oracle_fits()
    model = oracle_llama_model() if llama else None
    prompt, steps = (args.ref_prompt, args.ref_steps) if llama else (args.cpu_tokens, 8)
    for _ in range(args.warmup):
        oracle_sample(1, 16, 1, model)
    tot_tok, tot_s = 0, 0.0
    for _ in range(args.steps):
        tok, dt = oracle_sample(1, prompt, steps, model)
        tot_tok += tok
        tot_s += dt
    v = tot_tok / tot_s
    what = (f"Llama-2-7B-shaped workload (same model and exit law), bounded sample: its first {prompt} prompt tokens "
            f"+ {steps} generation steps per step") if llama else \
        (f"host memory below the fp64 Llama oracle's need: GPT-2-small workload, 1 prompt x {prompt} tokens + "
         f"{steps} generation steps per step")
    return {"metric": METRIC, "value": round(v, 3), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(tot_s / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": what},
            "cpu_baseline": {"value": round(v, 3), "unit": "tokens/s", "cores": cores(), "kind": "oracle",
                             "sample": what},
            "e2e": {"value": round(v, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def kernel_case_fill_small(device):
    """A small instance of the skipped-layer fill for kernel captures (ncu): Llama-7B layer
    shapes (D=4096, 32 heads x 128) but 8 layers and small FFN / HSM / vocabulary, 4096
    exited tokens at exit layer 4 (4 skipped layers): about 2 GB on the device, inputs
    and outputs larger than L2.  Three fills."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    cfg = synth.llama7b_config(n_layers=8, d_ffn=1024, vocab=1024, hsm_m1=512, hsm_m2=512, max_batch=4,
                               max_seq=1024, max_pass_tokens=64, block_shuffle_seed=7)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    adept.adept_seq_reserve(m.h, [cfg.max_seq] * 4)
    T = 4096
    h = synth.make_mapped_states(5, T, cfg.d_model, device=device)
    j = torch.arange(T, device=device, dtype=torch.int32)
    el = torch.full((T,), 4, dtype=torch.int32, device=device)
    for _ in range(3):
        adept.adept_skip_kv_fill(m.h, T, h, el, (j % 4).contiguous(), (j // 4).contiguous())
    m.check()
    torch.cuda.synchronize()
    print(json.dumps({"kernel_case": "fill_small", "T": T, "exit_layer": 4, "skipped_layers": 4, "ok": True}))
    m.close()


def kernel_case_fill_grid(device, grid_T, grid_i):
    """The skipped-layer fill grid alone (Llama-7B layers), one JSON line per cell."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    peaks, _ = load_peaks()
    for row in run_fill_micro(adept, device, peaks, grid_T, grid_i):
        print(json.dumps({"kernel_case": "fill_grid", **row}))


def kernel_case_llama_prefill(device):
    """Two early-exit prompt passes at the Llama-2-7B shape (2048 tokens, exits ~ N(24,4) on
    [8, 32]) for launch-list captures: the second pass is the one to capture."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    P = 2048
    cfg = synth.llama7b_config(max_batch=1, max_seq=P, max_pass_tokens=P)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    tok = synth.make_tokens(0, 1, P, cfg.vocab).to(device)
    fp = synth.forced_exits_truncnorm(0, P, 24.0, 4.0, 8, 32, name="forced_prompt").to(device)
    nxt = torch.empty(1, dtype=torch.int32, device=device)
    for _ in range(2):
        adept.adept_prefill(m.h, 1, P, tok.view(-1), 0.9, fp, None, None, nxt, None)
    torch.cuda.synchronize()
    m.check()
    print(json.dumps({"kernel_case": "llama_prefill", "prompt": P, "launches_per_pass": adept.adept_launch_count(m.h) // 2}))
    m.close()


def kernel_case_gpt2_decode(device):
    """The benchmark workload's prompt pass (8 x 512) and 8 generation steps (graph replay
    from the second), for launch-list captures of the generation step: the launches of
    one step are printed, the last steps are the ones to capture."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    cfg = workload_cfg()
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    tok = synth.make_tokens(0, B, P, cfg.vocab).to(device)
    fp = synth.forced_exits_uniform(0, B * P, LO, HI, name="forced_prompt").view(B, P).to(device)
    fd = synth.forced_exits_uniform(0, STEPS * B, LO, HI, name="forced_decode").view(STEPS, B).to(device)
    nxt = torch.empty(9, B, dtype=torch.int32, device=device)
    adept.adept_prefill(m.h, B, P, tok.view(-1), DELTA, fp.view(-1), None, None, nxt[0], None)
    adept.adept_launch_count(m.h)
    for s in range(8):
        adept.adept_decode_step(m.h, B, nxt[s], DELTA, fd[s], None, None, nxt[s + 1], None)
    torch.cuda.synchronize()
    m.check()
    print(json.dumps({"kernel_case": "gpt2_decode", "steps": 8, "launches_per_step": adept.adept_launch_count(m.h) // 8}))
    m.close()


def kernel_case_llama_decode_small(device):
    """Generation steps at Llama-2-7B layer shapes (D=4096, 32 heads x 128, SwiGLU 11008) with
    2 layers, a 1024-token vocabulary and a small HSM, batch 1, 64-token prompt, 4 steps:
    about 1 GB on the device; each layer's weights (404 MB) exceed L2, so the decode GEMMs'
    DRAM counters are meaningful in a kernel capture."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    cfg = synth.llama7b_config(n_layers=2, vocab=1024, hsm_m1=512, hsm_m2=512, max_batch=1, max_seq=128,
                               max_pass_tokens=64)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    tok = synth.make_tokens(0, 1, 64, cfg.vocab).to(device)
    nxt = torch.empty(5, 1, dtype=torch.int32, device=device)
    full = torch.full((64,), 2, dtype=torch.int32, device=device)
    adept.adept_prefill(m.h, 1, 64, tok.view(-1), DELTA, full, None, None, nxt[0], None)
    for s in range(4):
        adept.adept_decode_step(m.h, 1, nxt[s], DELTA, full[:1], None, None, nxt[s + 1], None)
    torch.cuda.synchronize()
    m.check()
    print(json.dumps({"kernel_case": "llama_decode_small", "steps": 4, "ok": True}))
    m.close()


def kernel_case_llama_decode_ctx(device):
    """Generation steps at Llama-2-7B layer shapes after the headline workload's 2048-token
    prompt (2 layers, a 1024-token vocabulary, a small HSM, batch 1, room for 2304 positions as
    in the headline: the attention grid of 32 heads x 18 key chunks), 3 steps: about 1 GB on the
    device."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    P = 2048
    cfg = synth.llama7b_config(n_layers=2, vocab=1024, hsm_m1=512, hsm_m2=512, max_batch=1, max_seq=P + 256,
                               max_pass_tokens=P)
    W = synth.make_weights(cfg, seed=0, device=device)
    m = adept.Model(cfg, W)
    del W
    tok = synth.make_tokens(0, 1, P, cfg.vocab).to(device)
    nxt = torch.empty(4, 1, dtype=torch.int32, device=device)
    full = torch.full((P,), 2, dtype=torch.int32, device=device)
    adept.adept_prefill(m.h, 1, P, tok.view(-1), DELTA, full, None, None, nxt[0], None)
    for s in range(3):
        adept.adept_decode_step(m.h, 1, nxt[s], DELTA, full[:1], None, None, nxt[s + 1], None)
    torch.cuda.synchronize()
    m.check()
    print(json.dumps({"kernel_case": "llama_decode_ctx", "prompt": P, "steps": 3, "ok": True}))
    m.close()


def kernel_case_hsm_train(device, n=8192, steps=2, shape="gpt2"):
    """HSM training steps at GPT-2-small shapes (the bench section's workload; about 5 GB on
    the device), Llama-2-7B shapes (about 25 GB) or BERT-base shapes (the encoder step, n / 128
    labelled rows): n examples, two steps after one warm-up."""
    import paper_2601_03700_gb300 as adept
    adept.load_library()
    if shape == "llama7b":
        cfg = synth.llama7b_config(n_layers=2, max_batch=1, max_seq=16)
    elif shape == "bert":
        cfg = synth.bert_base_config(n_layers=2, max_batch=1, max_seq=16)
    else:
        cfg = synth.gpt2_small_config(n_layers=2, max_batch=1, max_seq=16)
    W = synth.make_weights(cfg, seed=0)   # on the host: the launch list then holds the library's kernels only
    m = adept.Model(cfg, W)
    del W
    adept.adept_hsm_train_init(m.h, n)
    if shape == "bert":
        s_i, s_prev, inertia, s_fin, lab = [x.to(device) for x in synth.hsm_cls_batch(cfg, n, n // 128, seed=1)]
        step = lambda: adept.adept_hsm_train_step_cls(m.h, n, s_i, s_prev, inertia, s_fin, lab, 1e-4)  # noqa
    else:
        s_i, s_prev, inertia, tgt = [x.to(device) for x in synth.hsm_train_batch(cfg, n, seed=1)]
        step = lambda: adept.adept_hsm_train_step(m.h, n, s_i, s_prev, inertia, tgt, 1e-4)  # noqa
    for _ in range(steps + 1):
        step()
    torch.cuda.synchronize()
    m.check()
    print(json.dumps({"kernel_case": "hsm_train", "n": n, "steps": steps + 1, "ok": True}))
    m.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--kernel-case", default=None,
                    choices=["fill_small", "fill_grid", "llama_prefill", "gpt2_decode", "llama_decode_small",
                             "llama_decode_ctx", "hsm_train"])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-kv-fill", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-llama", action="store_true")
    ap.add_argument("--fill-T", default="1,4,16,64,256,1024,4096,16384,65536")
    ap.add_argument("--fill-i", default="4,8,16,24")
    ap.add_argument("--cpu-tokens", type=int, default=256, help="prompt tokens of the CPU-baseline oracle sample")
    ap.add_argument("--cpu-steps", type=int, default=8, help="generation steps of the CPU-baseline oracle sample")
    ap.add_argument("--ref-prompt", type=int, default=64, help="prompt tokens per step of --impl reference")
    ap.add_argument("--ref-steps", type=int, default=2, help="generation steps per step of --impl reference")
    ap.add_argument("--hsm-n", type=int, default=8192, help="examples per step of --kernel-case hsm_train")
    ap.add_argument("--hsm-shape", default="gpt2", choices=["gpt2", "llama7b", "bert"],
                    help="model shape of --kernel-case hsm_train")
    ap.add_argument("--oracle-sample", default=None, help="n_seq,prompt,steps: time the oracle alone (CPU)")
    args = ap.parse_args()
    if args.oracle_sample:
        n_seq, prompt, steps = (int(x) for x in args.oracle_sample.split(","))
        tok, dt = oracle_sample(n_seq, prompt, steps)
        print(json.dumps({"tokens": tok, "seconds": dt}), flush=True)
        return
    if args.kernel_case == "fill_small":
        kernel_case_fill_small(torch.device("cuda", 0))
        return
    if args.kernel_case == "fill_grid":
        kernel_case_fill_grid(torch.device("cuda", 0), [int(x) for x in args.fill_T.split(",")],
                              [int(x) for x in args.fill_i.split(",")])
        return
    if args.kernel_case == "llama_prefill":
        kernel_case_llama_prefill(torch.device("cuda", 0))
        return
    if args.kernel_case == "gpt2_decode":
        kernel_case_gpt2_decode(torch.device("cuda", 0))
        return
    if args.kernel_case == "llama_decode_small":
        kernel_case_llama_decode_small(torch.device("cuda", 0))
        return
    if args.kernel_case == "llama_decode_ctx":
        kernel_case_llama_decode_ctx(torch.device("cuda", 0))
        return
    if args.kernel_case == "hsm_train":
        kernel_case_hsm_train(torch.device("cuda", 0), n=args.hsm_n, shape=args.hsm_shape)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        line = reference_arm(args, rank, world)
        if line is not None:
            print(json.dumps(line), flush=True)
        return
    if world > 1:
        torch.cuda.set_device(local)
        torch.distributed.init_process_group("nccl")
    device = torch.device("cuda", torch.cuda.current_device())
    line = ours(args, rank, world, device)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
