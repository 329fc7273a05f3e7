"""Plain CPU oracle of ADEPT's token-level early-exit forward pass (float64 NumPy).

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct statement of
what the CUDA library computes.  Only the test suite, the smoke check and the
benchmark's CPU-baseline leg may import it; the library never does, and it shares
no code with the library (the two meet only through the seeded inputs of
``synth``).

What it follows (paper sections / equations / tables):

* Layers are 1-indexed, i in [1, N], tokens j in [1, M] (Sec. 3, state space).
* Inertia ``I_j = sum_{d=1}^{i-1} s_hat_{d,j}`` with ``s_hat = s / ||s||`` and the
  exit rule ``<s_hat_{i,j}, I_hat_j> >= delta`` (Sec. 4.1).
* The Hidden State Mapper (Sec. 4.2, App. B Table S1): the three inputs are
  RMS-normalised separately, stacked to (3, D_h), a 3x3 convolution with stride 1
  and padding (0, 1) gives one D_h row, then the 4-FC MLP with its normalisations
  and two additions.
* Skipped-layer K/V (Eq. 6, the decoupling of Sec. 4; Eq. 9, KV generation in Sec. 4.3):
  for every r > i*, the K/V of layer r are layer r's K/V projection of the mapped
  state s~_N, computed directly from s~_N (no sequential unfolding).
* Dynamic shrinkage (App. I): each layer runs only on the still-active tokens.
* Threshold calibration (Sec. 4.1, Sec. 5.1): bisection on delta to a target reduction
  in computation (RDC) over a calibration batch.
* Exit-rule variants (App. H.2-H.3): the local similarity cos(s_i, s_{i-1}), both
  similarities, and all-at-once prompt exits decided by each sequence's last token.
* Encoder "stop entirely" (Sec. 4.3, downstream tasks): exited tokens get no deeper K/V
  and drop out of deeper attention; their s~ feeds the classifier.
* Encoder-decoder models (Sec. 5.2, the OFA setting): the encoder runs its early-exit pass;
  its final states (s_N, or s~_N for exited tokens) are the source of every decoder layer's
  cross-attention; the decoder runs the same early-exit pass (its own HSM, skipped-layer
  K/V of its self-attention), each of its layers cross-attending after self-attention.

Readings where the paper is silent (each one is also listed in the design notes):

* No exit test at i = 1 (the inertia sum is empty) nor at i = N (full depth); a
  zero-norm state never exits.
* The similarity is computed on the residual-stream output of layer i (the
  post-LN output for the post-norm encoder).
* Layer r's K/V of an exited token apply layer r's own input norm, W_K / W_V,
  biases and RoPE at the token's position to s~_N -- exactly what layer r would do
  to an input s~_N.
* HSM activations: erf-GELU after FC1 and FC2; the MLP addition adds FC1's output,
  the final addition adds the convolution output.
* The HSM's inertia input is the sum *before* adding s_hat_i.
* Precision contract for bf16 models: weights are bf16 values; every GEMM input
  (activations), Q and the cached K/V are rounded to bf16 (round-to-nearest-even);
  everything else stays in float64 here.  fp32 models round nothing.
* Cross-attention sublayer (the paper names the encoder-decoder architecture but not its
  layer): pre-LN like the decoder's other sublayers, h <- h + W_Oc attn(LN_c(h) W_Qc, E W_Kc,
  E W_Vc) + b_Oc between self-attention and the FFN, over all source positions of the
  token's sequence (not causal); E are the encoder's final states, projected without a
  further norm.  An exited decoder token skips its deeper layers' cross-attention too; the
  source K/V depend on the encoder alone and need no fill.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, Optional

import numpy as np
from scipy.special import erf

LLAMA, GPT2, BERT = 0, 1, 2


# ----------------------------------------------------------------------------
# elementary pieces
# ----------------------------------------------------------------------------

def round_bf16(x) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even), returned as float64.

    The value goes through float32 first; the float32 -> bfloat16 step keeps the top
    16 bits after adding half an ulp (plus the tie-to-even bit).
    """
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def rms_normalize(x: np.ndarray, eps: float) -> np.ndarray:
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def rmsnorm(x, g, eps):
    return rms_normalize(x, eps) * g


def layernorm(x, g, b, eps):
    mu = np.mean(x, axis=-1, keepdims=True)
    var = np.mean((x - mu) ** 2, axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def gelu_erf(x):
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def silu(x):
    return x / (1.0 + np.exp(-x))


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing: feature i pairs with i + d/2.

    x: [n, heads, d]; pos: [n].  Frequency of pair i is theta^(-2i/d).
    """
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = pos.astype(np.float64)[:, None] * inv[None, :]          # [n, half]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def cosine(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Row-wise <a/|a|, b/|b|>; -inf where either norm is zero (never exits)."""
    na = np.linalg.norm(a, axis=-1)
    nb = np.linalg.norm(b, axis=-1)
    dot = np.sum(a * b, axis=-1)
    out = np.full(dot.shape, -np.inf)
    ok = (na > 0) & (nb > 0)
    out[ok] = dot[ok] / (na[ok] * nb[ok])
    return out


def unit(x: np.ndarray) -> np.ndarray:
    """s_hat = s / ||s|| (Sec. 4.1); a zero row stays zero."""
    n = np.linalg.norm(x, axis=-1, keepdims=True)
    return np.where(n > 0, x / np.where(n > 0, n, 1.0), 0.0)


def hsm_conv(X: np.ndarray, w: np.ndarray, b: float) -> np.ndarray:
    """Table S1 convolution: input (3, D) -> output (1, D), 3x3 kernel, stride 1,
    padding 0 rows / 1 column, zero padding, cross-correlation.

    X: [n, 3, D]; w: [3, 3] (row a, column offset u-1); returns [n, D].
    """
    n, three, D = X.shape
    Xp = np.zeros((n, three, D + 2))
    Xp[:, :, 1:D + 1] = X
    out = np.full((n, D), float(b))
    for a in range(3):
        for u in range(3):
            out += w[a, u] * Xp[:, a, u:u + D]
    return out


def hsm_param_count(d: int, m1: int, m2: int) -> int:
    """Weights of the four FC layers of Table S1 (biases, norms and the 9 conv taps excluded)."""
    return d * m1 + m1 * m2 + m2 * m1 + m1 * d


# ----------------------------------------------------------------------------
# model
# ----------------------------------------------------------------------------

class OracleModel:
    """Weights as float64 arrays plus the shape table (``synth.ModelConfig``)."""

    def __init__(self, cfg, weights: Dict[str, object]):
        self.cfg = cfg
        self.w = {}
        for k, v in weights.items():
            if hasattr(v, "detach"):
                v = v.detach().to("cpu").double().numpy()
            self.w[k] = np.asarray(v, dtype=np.float64)
        self.bf16 = cfg.dtype == "bf16"

    def rb(self, x):
        return round_bf16(x) if self.bf16 else x

    def L(self, i: int, name: str) -> np.ndarray:
        """Weight of paper layer i (1-based)."""
        return self.w[f"layers.{i - 1}.{name}"]

    def has(self, i: int, name: str) -> bool:
        return f"layers.{i - 1}.{name}" in self.w

    # -- the layer's input normalisation (pre-norm families; identity for the encoder)
    def attn_input(self, i: int, h: np.ndarray) -> np.ndarray:
        c = self.cfg
        if c.family == LLAMA:
            return rmsnorm(h, self.L(i, "attn_norm.g"), c.norm_eps)
        if c.family == GPT2:
            return layernorm(h, self.L(i, "attn_norm.g"), self.L(i, "attn_norm.b"), c.norm_eps)
        return h

    def _proj(self, x, i, wname, bname):
        y = x @ self.L(i, wname).T
        if self.has(i, bname):
            y = y + self.L(i, bname)
        return y

    def kv_project(self, i: int, h: np.ndarray, pos: np.ndarray):
        """Layer i's K and V of hidden states h (the layer's input) at positions pos.

        Used both for an active token's own layer input and, for an exited token, with
        h = s~_N (Sec. 4.3 KV generation).  Returns bf16-rounded [n, Hkv, dh] arrays.
        """
        c = self.cfg
        x = self.rb(self.attn_input(i, h))
        k = self._proj(x, i, "wk", "bk").reshape(len(h), c.n_kv_heads, c.head_dim)
        v = self._proj(x, i, "wv", "bv").reshape(len(h), c.n_kv_heads, c.head_dim)
        if c.family == LLAMA:
            k = rope(k, pos, c.rope_theta)
        return self.rb(k), self.rb(v)

    def q_project(self, i: int, h: np.ndarray, pos: np.ndarray):
        c = self.cfg
        x = self.rb(self.attn_input(i, h))
        q = self._proj(x, i, "wq", "bq").reshape(len(h), c.n_heads, c.head_dim)
        if c.family == LLAMA:
            q = rope(q, pos, c.rope_theta)
        return self.rb(q)

    # -- cross-attention (encoder-decoder decoders)
    def cross_q(self, i: int, h: np.ndarray):
        c = self.cfg
        x = self.rb(layernorm(h, self.L(i, "cross_norm.g"), self.L(i, "cross_norm.b"), c.norm_eps))
        return self.rb(self._proj(x, i, "cwq", "cbq").reshape(len(h), c.n_heads, c.head_dim))

    def cross_kv(self, i: int, e: np.ndarray):
        """Layer i's source K and V of encoder final states e [S, D]."""
        c = self.cfg
        x = self.rb(e)
        k = self._proj(x, i, "cwk", "cbk").reshape(len(e), c.n_kv_heads, c.head_dim)
        v = self._proj(x, i, "cwv", "cbv").reshape(len(e), c.n_kv_heads, c.head_dim)
        return self.rb(k), self.rb(v)

    def embed(self, tokens: np.ndarray, pos: np.ndarray) -> np.ndarray:
        c = self.cfg
        e = self.w["tok_emb"][tokens]
        if c.family == GPT2:
            e = e + self.w["pos_emb"][pos]
        elif c.family == BERT:
            e = layernorm(e + self.w["pos_emb"][pos] + self.w["type_emb"],
                          self.w["emb_ln.g"], self.w["emb_ln.b"], c.norm_eps)
        return e

    # -- Hidden State Mapper (Sec. 4.2, App. B Table S1)
    def hsm(self, s_i: np.ndarray, s_prev: np.ndarray, inertia: np.ndarray) -> np.ndarray:
        c, w, rb = self.cfg, self.w, self.rb
        eps = c.hsm_eps
        X = np.stack([rmsnorm(s_i, w["hsm.g0"], eps),
                      rmsnorm(s_prev, w["hsm.g0"], eps),
                      rmsnorm(inertia, w["hsm.g0"], eps)], axis=1)        # [n, 3, D]
        c0 = hsm_conv(X, w["hsm.conv_w"], w["hsm.conv_b"][0])              # [n, D]
        h1 = gelu_erf(rb(c0) @ w["hsm.fc1_w"].T + w["hsm.fc1_b"])          # [n, m1]
        h2 = gelu_erf(rb(h1) @ w["hsm.fc2_w"].T + w["hsm.fc2_b"])          # [n, m2]
        h3 = rb(h2) @ w["hsm.fc3_w"].T + w["hsm.fc3_b"]                    # [n, m1]
        h4 = rmsnorm(h3, w["hsm.g1"], eps) + h1                            # MLP add
        h5 = rb(h4) @ w["hsm.fc4_w"].T + w["hsm.fc4_b"]                    # [n, D]
        return rmsnorm(h5, w["hsm.g2"], eps) + c0                          # final add

    # -- output heads
    def lm_logits(self, x: np.ndarray) -> np.ndarray:
        c, w = self.cfg, self.w
        if c.family == LLAMA:
            return self.rb(rmsnorm(x, w["final_norm.g"], c.norm_eps)) @ w["lm_head"].T
        return self.rb(layernorm(x, w["final_norm.g"], w["final_norm.b"], c.norm_eps)) @ w["tok_emb"].T

    def cls_logits(self, x: np.ndarray) -> np.ndarray:
        w = self.w
        pooled = np.tanh(self.rb(x) @ w["pool.w"].T + w["pool.b"])
        return self.rb(pooled) @ w["cls.w"].T + w["cls.b"]


# ----------------------------------------------------------------------------
# KV cache (plain, contiguous per sequence; unwritten entries are NaN)
# ----------------------------------------------------------------------------

class OracleCache:
    def __init__(self, cfg, batch: int, max_seq: int):
        shape = (batch, max_seq, cfg.n_kv_heads, cfg.head_dim)
        self.K = [np.full(shape, np.nan) for _ in range(cfg.n_layers)]
        self.V = [np.full(shape, np.nan) for _ in range(cfg.n_layers)]
        self.lens = np.zeros(batch, dtype=np.int64)

    def write(self, i: int, seq, pos, k, v):
        self.K[i - 1][seq, pos] = k
        self.V[i - 1][seq, pos] = v


class CrossSource:
    """Every decoder layer's source K/V per sequence: K[i - 1][b] is [src_len[b], Hkv, dh]."""

    def __init__(self, m: "OracleModel", states):
        """states: per sequence b, the encoder's final states [src_len[b], D] (s_N of tokens
        that ran to full depth, s~_N of exited ones)."""
        self.src_len = np.array([len(e) for e in states], dtype=np.int64)
        self.K = [[None] * len(states) for _ in range(m.cfg.n_layers)]
        self.V = [[None] * len(states) for _ in range(m.cfg.n_layers)]
        for i in range(1, m.cfg.n_layers + 1):
            for b, e in enumerate(states):
                self.K[i - 1][b], self.V[i - 1][b] = m.cross_kv(i, np.asarray(e, dtype=np.float64))


def attend(m: OracleModel, q: np.ndarray, qpos: np.ndarray, K: np.ndarray, V: np.ndarray,
           causal: bool, key_mask: Optional[np.ndarray] = None) -> np.ndarray:
    """Softmax attention of one sequence's queries q [n, H, dh] over keys K/V [L, Hkv, dh].

    Causal: query at position p sees keys 0..p.  key_mask [L] (optional): only those keys.
    Returns [n, H*dh]."""
    c = m.cfg
    rep = c.n_heads // c.n_kv_heads
    if key_mask is not None:
        K, V = np.where(key_mask[:, None, None], K, 0.0), np.where(key_mask[:, None, None], V, 0.0)
    Kh = np.repeat(K, rep, axis=1)
    Vh = np.repeat(V, rep, axis=1)
    sc = np.einsum("nhd,lhd->hnl", q, Kh) / math.sqrt(c.head_dim)
    if causal:
        kpos = np.arange(K.shape[0])
        sc = np.where(kpos[None, None, :] <= qpos[None, :, None], sc, -np.inf)
    if key_mask is not None:
        sc = np.where(key_mask[None, None, :], sc, -np.inf)
    sc = sc - np.max(sc, axis=-1, keepdims=True)
    p = np.exp(sc)
    p = p / np.sum(p, axis=-1, keepdims=True)
    out = np.einsum("hnl,lhd->nhd", p, Vh)
    return out.reshape(q.shape[0], c.n_heads * c.head_dim)


def layer_body(m: OracleModel, i: int, h: np.ndarray, seq: np.ndarray, pos: np.ndarray,
               cache: OracleCache, causal: bool, kv_len: np.ndarray,
               key_active: Optional[Dict[int, np.ndarray]] = None,
               cross: Optional[CrossSource] = None) -> np.ndarray:
    """Everything of layer i after its K/V were cached: Q, attention, O, FFN, residuals.

    h: [n, D] layer inputs of the active tokens; returns their layer outputs.
    key_active (optional, "stop entirely"): per sequence, the positions whose K/V layer i
    holds; attention sees only those keys.
    cross (encoder-decoder decoders): the source K/V; the cross-attention sublayer runs
    between self-attention and the FFN."""
    c, rb = m.cfg, m.rb
    q = m.q_project(i, h, pos)
    att = np.zeros((len(h), c.n_heads * c.head_dim))
    for b in np.unique(seq):
        sel = np.nonzero(seq == b)[0]
        L = int(kv_len[b])
        km = None if key_active is None else key_active[int(b)][:L]
        att[sel] = attend(m, q[sel], pos[sel], cache.K[i - 1][b, :L], cache.V[i - 1][b, :L], causal, km)
    o = rb(att) @ m.L(i, "wo").T
    if m.has(i, "bo"):
        o = o + m.L(i, "bo")
    if c.family == BERT:
        h1 = layernorm(h + o, m.L(i, "attn_norm.g"), m.L(i, "attn_norm.b"), c.norm_eps)
        f = rb(gelu_erf(rb(h1) @ m.L(i, "w_fc").T + m.L(i, "b_fc")))
        f = f @ m.L(i, "w_proj").T + m.L(i, "b_proj")
        return layernorm(h1 + f, m.L(i, "ffn_norm.g"), m.L(i, "ffn_norm.b"), c.norm_eps)
    h1 = h + o
    if cross is not None:
        qc = m.cross_q(i, h1)
        ac = np.zeros((len(h), c.n_heads * c.head_dim))
        for b in np.unique(seq):
            sel = np.nonzero(seq == b)[0]
            ac[sel] = attend(m, qc[sel], pos[sel], cross.K[i - 1][b], cross.V[i - 1][b], False)
        h1 = h1 + rb(ac) @ m.L(i, "cwo").T + m.L(i, "cbo")
    if c.family == GPT2:
        x = rb(layernorm(h1, m.L(i, "ffn_norm.g"), m.L(i, "ffn_norm.b"), c.norm_eps))
        f = rb(gelu_tanh(x @ m.L(i, "w_fc").T + m.L(i, "b_fc")))
        return h1 + f @ m.L(i, "w_proj").T + m.L(i, "b_proj")
    x = rb(rmsnorm(h1, m.L(i, "ffn_norm.g"), c.norm_eps))
    f = rb(silu(x @ m.L(i, "w_gate").T) * (x @ m.L(i, "w_up").T))
    return h1 + f @ m.L(i, "w_down").T


# ----------------------------------------------------------------------------
# the early-exit pass (App. I process, Sec. 4.1-4.3 pieces)
# ----------------------------------------------------------------------------

@dataclass
class PassResult:
    exit_layer: np.ndarray      # [T] int, 1..N (N = full depth)
    sim: np.ndarray             # [T, N] cosine at each tested layer, NaN elsewhere
    final: np.ndarray           # [T, D] s~_N of exited tokens, s_N of the rest
    logits: Optional[np.ndarray] = None
    next_token: Optional[np.ndarray] = None


def check_forced(forced: np.ndarray, n_layers: int):
    bad = (forced != 0) & ((forced < 2) | (forced > n_layers))
    if np.any(bad):
        raise ValueError("forced exit layers must be 0 (threshold) or in [2, N]")


def early_exit_pass(m: OracleModel, cache: OracleCache, s0: np.ndarray, seq: np.ndarray,
                    pos: np.ndarray, delta: float, forced: Optional[np.ndarray], causal: bool,
                    kv_len: np.ndarray, hsm_mode: str = "hsm", metric: str = "global",
                    aao_len: int = 0, stop_entirely: bool = False,
                    cross: Optional[CrossSource] = None) -> PassResult:
    """Run tokens (all in parallel, App. I) through layers 1..N with token-level exits.

    For each layer i: (a) K/V of the active tokens from their layer input go to the
    cache; (b) the rest of the layer runs for the active tokens; (c) for 2 <= i <= N-1
    the exit test <s_hat_i, I_hat> >= delta (or i == forced exit layer); (d) the
    inertia takes s_hat_i; (e) each exiting token is mapped by the HSM and its K/V of
    every skipped layer r > i are produced from s~_N at once.

    Variants (App. H.3, "Local vs Global Metric"; App. H.2, "All-at-Once Early-Exit"):
    metric "local" tests cos(s_i, s_{i-1}) (s_{i-1} = the layer's input), "both" requires
    the global and the local similarity to reach delta (the recorded similarity is then
    their minimum); aao_len = P > 0 (prompt passes) makes every token take the decision of
    its sequence's last prompt token (position P - 1), so a sequence leaves at once.
    stop_entirely (encoders, Sec. 4.3 on downstream tasks: computation stops beyond the exit
    layer): an exiting token gets s~ for the classifier but no K/V of deeper layers, and the
    attention of a deeper layer sees only the tokens still active there.
    cross (encoder-decoder decoders): the source K/V of every layer's cross-attention.
    """
    if metric not in ("global", "local", "both"):
        raise ValueError(metric)
    c = m.cfg
    if (cross is not None) != (getattr(c, "max_src", 0) > 0):
        raise ValueError("cross-attention models take a CrossSource, other models none")
    N, T = c.n_layers, len(s0)
    forced = np.zeros(T, dtype=np.int64) if forced is None else np.asarray(forced, dtype=np.int64)
    check_forced(forced, N)
    s = s0.copy()
    inertia = np.zeros_like(s0)
    active = np.ones(T, dtype=bool)
    exit_layer = np.full(T, N, dtype=np.int64)
    sim = np.full((T, N), np.nan)
    final = np.zeros_like(s0)
    for i in range(1, N + 1):
        A = np.nonzero(active)[0]
        if len(A) == 0:
            break
        k, v = m.kv_project(i, s[A], pos[A])                              # (a)
        cache.write(i, seq[A], pos[A], k, v)
        key_active = None
        if stop_entirely:
            key_active = {int(b): np.zeros(int(kv_len[b]), dtype=bool) for b in np.unique(seq)}
            for j in A:
                key_active[int(seq[j])][int(pos[j])] = True
        s_new = layer_body(m, i, s[A], seq[A], pos[A], cache, causal, kv_len, key_active, cross)   # (b)
        exits = np.zeros(len(A), dtype=bool)
        if 2 <= i <= N - 1:                                                # (c)
            cg = cosine(s_new, inertia[A])
            cl = cosine(s_new, s[A])
            cs = cg if metric == "global" else cl if metric == "local" else np.minimum(cg, cl)
            sim[A, i - 1] = cs
            f = forced[A]
            exits = np.where(f > 0, f == i, cs >= delta)
            if aao_len:
                last = {int(seq[j]): bool(exits[k]) for k, j in enumerate(A) if pos[j] == aao_len - 1}
                exits = np.array([last[int(seq[j])] for j in A], dtype=bool)
        I_before = inertia[A]
        inertia[A] = I_before + unit(s_new)                                # (d)
        E = A[exits]
        if len(E):                                                          # (e)
            if hsm_mode == "hsm":
                st = m.hsm(s_new[exits], s[E], I_before[exits])
            elif hsm_mode == "identity":
                st = s_new[exits].copy()
            else:
                raise ValueError(hsm_mode)
            final[E] = st
            exit_layer[E] = i
            for r in range(i + 1, N + 1) if not stop_entirely else ():
                kr, vr = m.kv_project(r, st, pos[E])
                cache.write(r, seq[E], pos[E], kr, vr)
        s[A] = s_new
        active[E] = False
    final[active] = s[active]
    return PassResult(exit_layer=exit_layer, sim=sim, final=final)


def prefill(m: OracleModel, cache: OracleCache, tokens: np.ndarray, delta: float,
            forced: Optional[np.ndarray] = None, hsm_mode: str = "hsm", metric: str = "global",
            all_at_once: bool = False, stop_entirely: bool = False,
            cross: Optional[CrossSource] = None) -> PassResult:
    """Prompt pass for sequences 0..B-1 (resets them); tokens [B, P].

    Decoder: logits [B, V] of each sequence's last position and its greedy token
    (lowest index on ties).  Encoder: bidirectional attention; classifier logits
    [B, C] from position 0's final state."""
    c = m.cfg
    if stop_entirely and c.family != BERT:
        raise ValueError("the stop-entirely variant is defined for encoders")
    tokens = np.asarray(tokens)
    B, P = tokens.shape
    seq = np.repeat(np.arange(B), P)
    pos = np.tile(np.arange(P), B)
    for l in range(c.n_layers):
        cache.K[l][:B] = np.nan
        cache.V[l][:B] = np.nan
    cache.lens[:B] = P
    s0 = m.embed(tokens.reshape(-1), pos)
    causal = c.family != BERT
    kv_len = cache.lens.copy()
    res = early_exit_pass(m, cache, s0, seq, pos, delta,
                          None if forced is None else np.asarray(forced).reshape(-1),
                          causal, kv_len, hsm_mode, metric, P if all_at_once else 0, stop_entirely, cross)
    fin = res.final.reshape(B, P, -1)
    if c.family == BERT:
        res.logits = m.cls_logits(fin[:, 0])
    else:
        res.logits = m.lm_logits(fin[:, P - 1])
        res.next_token = np.argmax(res.logits, axis=-1)
    return res


def decode_step(m: OracleModel, cache: OracleCache, tokens: np.ndarray, delta: float,
                forced: Optional[np.ndarray] = None, hsm_mode: str = "hsm", metric: str = "global",
                cross: Optional[CrossSource] = None) -> PassResult:
    """One generation step: token b of sequence b at position lens[b] (App. I, generation)."""
    c = m.cfg
    if c.family == BERT:
        raise ValueError("decode is defined for decoder models only")
    tokens = np.asarray(tokens).reshape(-1)
    B = len(tokens)
    seq = np.arange(B)
    pos = cache.lens[:B].copy()
    cache.lens[:B] += 1
    kv_len = cache.lens.copy()
    s0 = m.embed(tokens, pos)
    res = early_exit_pass(m, cache, s0, seq, pos, delta,
                          None if forced is None else np.asarray(forced).reshape(-1),
                          True, kv_len, hsm_mode, metric, cross=cross)
    res.logits = m.lm_logits(res.final)
    res.next_token = np.argmax(res.logits, axis=-1)
    return res


def reduction_in_computation(exit_layer: np.ndarray, n_layers: int) -> float:
    """RDC, the reduction in computation the paper reports (Sec. 5.1, Tables 3-5): the
    fraction of the T x N layer evaluations of a pass that early exit skips,
    1 - (sum_j depth_j) / (T N), where depth_j = i*_j is token j's exit layer."""
    e = np.asarray(exit_layer, dtype=np.float64).reshape(-1)
    return 1.0 - float(np.sum(e)) / (len(e) * n_layers)


def calibrate_threshold(m: OracleModel, tokens: np.ndarray, target_rdc: float, lo: float = -1.0,
                        hi: float = 1.0, max_iter: int = 24, tol: float = 0.005, hsm_mode: str = "hsm"):
    """Threshold calibration (Sec. 4.1: delta is set to meet the computation budget
    C_threshold; Sec. 5.1): bisection on delta over the prompt pass of a calibration
    batch until its RDC is within tol of target_rdc.

    A higher delta asks for a closer alignment before a token may leave, so fewer tokens
    leave and the RDC falls: when the batch's RDC is above the target, the threshold
    moves up (lo = delta), otherwise down (hi = delta).  The midpoints are dyadic
    fractions of [lo, hi], exact in float32 for the first 24 steps.  Returns
    (delta, rdc, [(delta, rdc) of every pass])."""
    tokens = np.asarray(tokens)
    B, P = tokens.shape
    N = m.cfg.n_layers
    hist = []
    delta = rdc = None
    for _ in range(max_iter):
        delta = 0.5 * (lo + hi)
        cache = OracleCache(m.cfg, B, P)
        res = prefill(m, cache, tokens, delta, hsm_mode=hsm_mode)
        rdc = reduction_in_computation(res.exit_layer, N)
        hist.append((delta, rdc))
        if abs(rdc - target_rdc) <= tol:
            break
        if rdc > target_rdc:
            lo = delta
        else:
            hi = delta
    return delta, rdc, hist


def skip_kv_fill(m: OracleModel, mapped: np.ndarray, exit_layer: np.ndarray, pos: np.ndarray):
    """K/V of every skipped layer r > i*_j for mapped states s~_N (Sec. 4.3).

    Returns {r: (K [n_r, Hkv, dh], V, token indices)} for r = 2..N."""
    N = m.cfg.n_layers
    out = {}
    for r in range(2, N + 1):
        sel = np.nonzero(exit_layer < r)[0]
        if len(sel) == 0:
            continue
        k, v = m.kv_project(r, mapped[sel], pos[sel])
        out[r] = (k, v, sel)
    return out
