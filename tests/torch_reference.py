"""An independent float64 reference built from torch.nn.functional library routines.

Used only to pin the oracle: it evaluates the same definitions in a different order
(one token at a time, all layers of a token before the next token -- the
"sequential unfold"), with library kernels (F.linear, F.rms_norm, F.layer_norm,
F.conv2d, F.scaled_dot_product_attention, complex-number RoPE) instead of the
oracle's NumPy expressions.  Layers are 1-based as in the paper.

bf16=True states the bf16 precision contract on its own: weights are bf16 values, and
torch's own float -> bfloat16 cast (round to nearest even) is applied to every GEMM input
(the normalised layer and head inputs, the attention output, the FFN's activated hidden
rows, the mapper's FC inputs, the pooler's input and output, the encoder states of the
cross-attention's K/V projection), to Q and to the cached K and V (self- and cross-
attention); everything else stays float64.
"""
from __future__ import annotations

import math

import torch
import torch.nn.functional as F

LLAMA, GPT2, BERT = 0, 1, 2


class TorchRef:
    def __init__(self, cfg, W, bf16: bool = False):
        self.c = cfg
        self.W = {k: (v if torch.is_tensor(v) else torch.as_tensor(v)).double() for k, v in W.items()}
        self.bf16 = bf16

    def r(self, x):
        """A contract rounding point: bf16 round trip in bf16 mode, identity otherwise."""
        return x.to(torch.bfloat16).double() if self.bf16 else x

    def lw(self, i, n):
        return self.W.get(f"layers.{i - 1}.{n}")

    # ---------------------------------------------------------------- pieces
    def rope(self, x, pos):
        """x [..., H, d] at positions pos [...]: pairs (k, k + d/2) as complex numbers."""
        d = x.shape[-1]
        half = d // 2
        freqs = self.c.rope_theta ** (-torch.arange(0, half, dtype=torch.float64) * 2.0 / d)
        ang = pos.double()[..., None] * freqs                           # [..., half]
        rot = torch.polar(torch.ones_like(ang), ang)[..., None, :]      # [..., 1, half]
        z = torch.complex(x[..., :half], x[..., half:]) * rot
        return torch.cat([z.real, z.imag], dim=-1)

    def pre_attn(self, i, h):
        c = self.c
        if c.family == LLAMA:
            return F.rms_norm(h, (c.d_model,), self.lw(i, "attn_norm.g"), c.norm_eps)
        if c.family == GPT2:
            return F.layer_norm(h, (c.d_model,), self.lw(i, "attn_norm.g"), self.lw(i, "attn_norm.b"), c.norm_eps)
        return h

    def kv(self, i, h, pos):
        c = self.c
        x = self.r(self.pre_attn(i, h))
        k = F.linear(x, self.lw(i, "wk"), self.lw(i, "bk")).unflatten(-1, (c.n_kv_heads, c.head_dim))
        v = F.linear(x, self.lw(i, "wv"), self.lw(i, "bv")).unflatten(-1, (c.n_kv_heads, c.head_dim))
        if c.family == LLAMA:
            k = self.rope(k, pos)
        return self.r(k), self.r(v)

    def q(self, i, h, pos):
        c = self.c
        x = self.r(self.pre_attn(i, h))
        q = F.linear(x, self.lw(i, "wq"), self.lw(i, "bq")).unflatten(-1, (c.n_heads, c.head_dim))
        if c.family == LLAMA:
            q = self.rope(q, pos)
        return self.r(q)

    # ---------------------------------------------------------------- cross-attention
    def cross_kv(self, i, e):
        """Layer i's source K, V [S, Hkv, dh] of encoder final states e [S, D]."""
        c = self.c
        x = self.r(e)
        k = F.linear(x, self.lw(i, "cwk"), self.lw(i, "cbk")).unflatten(-1, (c.n_kv_heads, c.head_dim))
        v = F.linear(x, self.lw(i, "cwv"), self.lw(i, "cbv")).unflatten(-1, (c.n_kv_heads, c.head_dim))
        return self.r(k), self.r(v)

    def cross_sublayer(self, i, h1, src):
        """h1 [..., D] of one sequence + its cross-attention over src = (K, V) [S, Hkv, dh]."""
        c, r = self.c, self.r
        x = r(F.layer_norm(h1, (c.d_model,), self.lw(i, "cross_norm.g"), self.lw(i, "cross_norm.b"), c.norm_eps))
        q = r(F.linear(x, self.lw(i, "cwq"), self.lw(i, "cbq")).unflatten(-1, (c.n_heads, c.head_dim)))
        rep = c.n_heads // c.n_kv_heads
        k = src[0].repeat_interleave(rep, dim=1).transpose(0, 1)        # [H, S, dh]
        v = src[1].repeat_interleave(rep, dim=1).transpose(0, 1)
        qh = q.reshape(-1, c.n_heads, c.head_dim).transpose(0, 1)       # [H, n, dh]
        a = F.scaled_dot_product_attention(qh, k, v).transpose(0, 1).reshape(*h1.shape[:-1], -1)
        return h1 + F.linear(r(a), self.lw(i, "cwo"), self.lw(i, "cbo"))

    def after_attn(self, i, h, a, src=None):
        """Residual / FFN part of layer i given the attention output a [..., H*dh]; src: the
        sequence's source K/V of layer i (encoder-decoder decoders)."""
        c, r = self.c, self.r
        o = F.linear(r(a), self.lw(i, "wo"), self.lw(i, "bo"))
        if c.family == BERT:
            h1 = F.layer_norm(h + o, (c.d_model,), self.lw(i, "attn_norm.g"), self.lw(i, "attn_norm.b"), c.norm_eps)
            f = F.linear(r(F.gelu(F.linear(r(h1), self.lw(i, "w_fc"), self.lw(i, "b_fc")))),
                         self.lw(i, "w_proj"), self.lw(i, "b_proj"))
            return F.layer_norm(h1 + f, (c.d_model,), self.lw(i, "ffn_norm.g"), self.lw(i, "ffn_norm.b"), c.norm_eps)
        h1 = h + o
        if src is not None:
            h1 = self.cross_sublayer(i, h1, src)
        if c.family == GPT2:
            x = r(F.layer_norm(h1, (c.d_model,), self.lw(i, "ffn_norm.g"), self.lw(i, "ffn_norm.b"), c.norm_eps))
            f = r(F.gelu(F.linear(x, self.lw(i, "w_fc"), self.lw(i, "b_fc")), approximate="tanh"))
            return h1 + F.linear(f, self.lw(i, "w_proj"), self.lw(i, "b_proj"))
        x = r(F.rms_norm(h1, (c.d_model,), self.lw(i, "ffn_norm.g"), c.norm_eps))
        f = r(F.silu(F.linear(x, self.lw(i, "w_gate"))) * F.linear(x, self.lw(i, "w_up")))
        return h1 + F.linear(f, self.lw(i, "w_down"))

    def embed(self, tok, pos):
        c, W = self.c, self.W
        e = W["tok_emb"][tok]
        if c.family == GPT2:
            e = e + W["pos_emb"][pos]
        elif c.family == BERT:
            e = F.layer_norm(e + W["pos_emb"][pos] + W["type_emb"], (c.d_model,), W["emb_ln.g"],
                             W["emb_ln.b"], c.norm_eps)
        return e

    def hsm(self, s_i, s_prev, inertia):
        c, W = self.c, self.W
        D, eps = c.d_model, c.hsm_eps
        X = torch.stack([F.rms_norm(t, (D,), W["hsm.g0"], eps) for t in (s_i, s_prev, inertia)], 0)
        r = self.r
        c0 = F.conv2d(X[None, None], W["hsm.conv_w"][None, None], W["hsm.conv_b"], stride=1,
                      padding=(0, 1))[0, 0, 0]
        h1 = F.gelu(F.linear(r(c0), W["hsm.fc1_w"], W["hsm.fc1_b"]))
        h2 = F.gelu(F.linear(r(h1), W["hsm.fc2_w"], W["hsm.fc2_b"]))
        h3 = F.linear(r(h2), W["hsm.fc3_w"], W["hsm.fc3_b"])
        h4 = F.rms_norm(h3, (c.hsm_m1,), W["hsm.g1"], eps) + h1
        h5 = F.linear(r(h4), W["hsm.fc4_w"], W["hsm.fc4_b"])
        return F.rms_norm(h5, (D,), W["hsm.g2"], eps) + c0

    def head(self, x):
        c, W, r = self.c, self.W, self.r
        if c.family == LLAMA:
            return F.linear(r(F.rms_norm(x, (c.d_model,), W["final_norm.g"], c.norm_eps)), W["lm_head"])
        if c.family == GPT2:
            return F.linear(r(F.layer_norm(x, (c.d_model,), W["final_norm.g"], W["final_norm.b"], c.norm_eps)),
                            W["tok_emb"])
        pooled = torch.tanh(F.linear(r(x), W["pool.w"], W["pool.b"]))
        return F.linear(r(pooled), W["cls.w"], W["cls.b"])

    # ---------------------------------------------------------------- full depth, batched
    def full_forward(self, tokens, source=None):
        """Standard full-depth forward of [B, P] tokens with SDPA; no cache.  source
        (encoder-decoder decoders): per sequence, the encoder's final states [S_b, D].

        Returns final hidden states [B, P, D]."""
        c = self.c
        tokens = torch.as_tensor(tokens)
        B, P = tokens.shape
        pos = torch.arange(P).expand(B, P)
        h = self.embed(tokens, pos)
        for i in range(1, c.n_layers + 1):
            q = self.q(i, h, pos).transpose(1, 2)
            k, v = self.kv(i, h, pos)
            rep = c.n_heads // c.n_kv_heads
            k = k.repeat_interleave(rep, dim=2).transpose(1, 2)
            v = v.repeat_interleave(rep, dim=2).transpose(1, 2)
            a = F.scaled_dot_product_attention(q, k, v, is_causal=c.family != BERT).transpose(1, 2).flatten(-2)
            if source is None:
                h = self.after_attn(i, h, a)
            else:
                h = torch.stack([self.after_attn(i, h[b], a[b], self.cross_kv(i, torch.as_tensor(source[b]).double()))
                                 for b in range(B)])
        return h

    # ---------------------------------------------------------------- token-major unfold
    def token_major(self, tokens, forced, hsm_mode="hsm", source=None):
        """One sequence, one token at a time, each token through all of its layers before
        the next token starts.  forced[j] in [2, N] is token j's exit layer (N = none).
        source (encoder-decoder decoders): the sequence's encoder final states [S, D].

        Returns (final [P, D], exit_layer [P], K dict, V dict) with K[i][j] the cached key
        of position j at layer i."""
        c = self.c
        src = None if source is None else {i: self.cross_kv(i, torch.as_tensor(source).double())
                                           for i in range(1, c.n_layers + 1)}
        N = c.n_layers
        tokens = torch.as_tensor(tokens).reshape(-1)
        P = len(tokens)
        K = {i: {} for i in range(1, N + 1)}
        V = {i: {} for i in range(1, N + 1)}
        final = torch.zeros(P, c.d_model, dtype=torch.float64)
        exit_layer = torch.full((P,), N, dtype=torch.int64)
        for j in range(P):
            pj = torch.tensor(j)
            h = self.embed(tokens[j], pj)
            inertia = torch.zeros(c.d_model, dtype=torch.float64)
            for i in range(1, N + 1):
                k, v = self.kv(i, h, pj)
                K[i][j], V[i][j] = k, v
                q = self.q(i, h, pj)                                       # [H, dh]
                keys = torch.stack([K[i][t] for t in range(j + 1)])          # [j+1, Hkv, dh]
                vals = torch.stack([V[i][t] for t in range(j + 1)])
                rep = c.n_heads // c.n_kv_heads
                keys = keys.repeat_interleave(rep, dim=1)
                vals = vals.repeat_interleave(rep, dim=1)
                w = torch.softmax(torch.einsum("hd,thd->ht", q, keys) / math.sqrt(c.head_dim), dim=-1)
                a = torch.einsum("ht,thd->hd", w, vals).reshape(-1)
                h_new = self.after_attn(i, h, a, None if src is None else src[i])
                leave = 2 <= i <= N - 1 and int(forced[j]) == i
                if leave:
                    st = self.hsm(h_new, h, inertia) if hsm_mode == "hsm" else h_new
                    final[j] = st
                    exit_layer[j] = i
                    for r in range(i + 1, N + 1):
                        K[r][j], V[r][j] = self.kv(r, st, pj)
                    break
                inertia = inertia + h_new / torch.linalg.vector_norm(h_new)
                h = h_new
            else:
                final[j] = h
        return final, exit_layer, K, V
