"""Seeded synthetic workloads: model shapes, weights, prompts and forced-exit laws.

This module is the one piece of code shared by the CPU oracle and the CUDA
library's tests and benchmark.  It holds *no* arithmetic of the method itself:
only shape tables and a counter-based random generator, so either side can
regenerate any tensor independently (a single weight matrix of a 7B-shaped
model can be rebuilt on the host without materialising the rest).

Generator definition (fixed; both the CPU and the CUDA builds of a tensor use
these exact integer operations, so the values agree bit for bit):

* ``key(seed, stream) = mix(mix(seed + G) ^ stream)`` where ``G`` is the
  splitmix64 increment 0x9E3779B97F4A7C15 and ``mix`` is the splitmix64
  finaliser (Steele, Lea, Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014).
* word ``i`` of the stream is ``mix(key + (i + 1) * G)`` (64-bit wrap-around).
* a uniform on [0, 1) is the top 53 bits of a word times 2^-53.
* a standard normal uses the Box-Muller transform on the uniforms drawn from
  words 2k and 2k+1, evaluated in float64 and only then rounded to the storage
  dtype (float32 or bfloat16, round-to-nearest-even).

``stream`` is a 32-bit CRC of the tensor's name, so the tensors of a model are
independent streams of one seed.
"""
from __future__ import annotations

import dataclasses
import math
import zlib
from typing import Dict, Optional

import torch

_MASK64 = (1 << 64) - 1
_G = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB


def _s64(v: int) -> int:
    """Python int (mod 2^64) -> the signed int64 with the same bits."""
    v &= _MASK64
    return v - (1 << 64) if v >= (1 << 63) else v


def _mix_int(z: int) -> int:
    z &= _MASK64
    z = ((z ^ (z >> 30)) * _M1) & _MASK64
    z = ((z ^ (z >> 27)) * _M2) & _MASK64
    return z ^ (z >> 31)


def _srl(x: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of an int64 tensor."""
    return (x >> k) & ((1 << (64 - k)) - 1)


def _mix(z: torch.Tensor) -> torch.Tensor:
    z = (z ^ _srl(z, 30)) * _s64(_M1)
    z = (z ^ _srl(z, 27)) * _s64(_M2)
    return z ^ _srl(z, 31)


def stream_id(name: str) -> int:
    return zlib.crc32(name.encode("utf-8")) & 0xFFFFFFFF


def stream_key(seed: int, name: str) -> int:
    return _mix_int(_mix_int(seed + _G) ^ stream_id(name))


def _words(key: int, start: int, count: int, device) -> torch.Tensor:
    i = torch.arange(start + 1, start + count + 1, dtype=torch.int64, device=device)
    return _mix(i * _s64(_G) + _s64(key))


def uniform(seed: int, name: str, n: int, device="cpu") -> torch.Tensor:
    """n float64 uniforms on [0, 1)."""
    w = _words(stream_key(seed, name), 0, n, device)
    return _srl(w, 11).to(torch.float64) * (2.0 ** -53)


_CHUNK = 1 << 24


def normal(seed: int, name: str, shape, std: float = 1.0, mean: float = 0.0,
           dtype=torch.float32, device="cpu") -> torch.Tensor:
    """Counter-based N(mean, std^2) tensor, rounded once to ``dtype``."""
    n = 1
    for s in shape:
        n *= int(s)
    key = stream_key(seed, name)
    out = torch.empty(n, dtype=dtype, device=device)
    for c0 in range(0, n, _CHUNK):
        c = min(_CHUNK, n - c0)
        w = _words(key, 2 * c0, 2 * c, device).view(c, 2)
        u1 = (_srl(w[:, 0], 11).to(torch.float64) + 1.0) * (2.0 ** -53)
        u2 = _srl(w[:, 1], 11).to(torch.float64) * (2.0 ** -53)
        z = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos((2.0 * math.pi) * u2)
        out[c0:c0 + c] = (z * std + mean).to(dtype)
    return out.view(*[int(s) for s in shape])


def randint(seed: int, name: str, n: int, lo: int, hi: int) -> torch.Tensor:
    """n int32 values uniform on the integers [lo, hi] (host)."""
    u = uniform(seed, name, n)
    return (torch.floor(u * (hi - lo + 1)).to(torch.int64) + lo).to(torch.int32)


# ----------------------------------------------------------------------------
# model shapes
# ----------------------------------------------------------------------------

LLAMA, GPT2, BERT = 0, 1, 2
FAMILY_NAMES = {LLAMA: "llama", GPT2: "gpt2", BERT: "bert"}


@dataclasses.dataclass
class ModelConfig:
    family: int
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    max_pos: int = 0           # learned positions (GPT-2 / BERT); 0 for RoPE models
    n_classes: int = 0         # encoder classifier outputs
    dtype: str = "bf16"        # "f32" or "bf16": storage and GEMM-input precision
    norm_eps: float = 1e-5
    rope_theta: float = 10000.0
    hsm_eps: float = 1e-6
    hsm_m1: int = 0            # HSM widths (FC1 out / FC2 out); 0 -> Table S1 (4D, 8D)
    hsm_m2: int = 0
    kv_block_tokens: int = 16
    max_batch: int = 8
    max_seq: int = 1024
    n_kv_heads: int = 0        # 0 -> n_heads
    kv_pool_blocks: int = 0    # 0 -> max_batch * ceil(max_seq / kv_block_tokens)
    max_pass_tokens: int = 0   # rows of per-pass workspaces; 0 -> max_batch * max_seq
    block_shuffle_seed: int = 0  # 0: KV blocks handed out in order; else a seeded permutation
    max_src: int = 0           # > 0 (GPT-2-family decoders): cross-attention over up to max_src
                               # encoder states per sequence (encoder-decoder models)

    def __post_init__(self):
        if self.n_kv_heads == 0:
            self.n_kv_heads = self.n_heads
        if self.hsm_m1 == 0:
            self.hsm_m1 = 4 * self.d_model
        if self.hsm_m2 == 0:
            self.hsm_m2 = 8 * self.d_model

    @property
    def d_q(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def d_kv(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32


def tiny_config(**kw) -> ModelConfig:
    """Tiny decoder: 4 layers, D=256, 4 heads, SwiGLU 1024, vocab 1024, fp32."""
    base = dict(family=LLAMA, n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ffn=1024,
                vocab=1024, dtype="f32", max_batch=4, max_seq=128)
    base.update(kw)
    return ModelConfig(**base)


def gpt2_small_config(**kw) -> ModelConfig:
    """GPT-2-small shape: 12 layers, D=768, 12 heads, GELU FFN 3072, vocab 50257, bf16."""
    base = dict(family=GPT2, n_layers=12, d_model=768, n_heads=12, head_dim=64, d_ffn=3072,
                vocab=50257, max_pos=1024, dtype="bf16", max_batch=8, max_seq=1024)
    base.update(kw)
    return ModelConfig(**base)


def llama7b_config(**kw) -> ModelConfig:
    """Llama-2-7B shape: 32 layers, D=4096, 32 heads x 128, SwiGLU 11008, vocab 32000.

    HSM widths (2D, 8D): 2*m1*D + 2*m1*m2 = 36 D^2 = 604M weights for D=4096.
    """
    base = dict(family=LLAMA, n_layers=32, d_model=4096, n_heads=32, head_dim=128, d_ffn=11008,
                vocab=32000, dtype="bf16", hsm_m1=2 * 4096, hsm_m2=8 * 4096, max_batch=1,
                max_seq=2304)
    base.update(kw)
    return ModelConfig(**base)


def ofa_base_configs(src_len: int = 256, tgt_len: int = 32, batch: int = 8, **kw):
    """OFA-base-shaped encoder-decoder (6 + 6 layers, D=768, 12 heads, GELU FFN 3072, BPE
    vocabulary 50265, bf16): a post-LN encoder with a 3-way classifier head (unused by the
    decoder) and a pre-LN decoder whose layers cross-attend to the encoder's final states.
    Returns (encoder config, decoder config)."""
    enc = dict(family=BERT, n_layers=6, d_model=768, n_heads=12, head_dim=64, d_ffn=3072, vocab=50265,
               max_pos=1024, n_classes=3, dtype="bf16", norm_eps=1e-5, max_batch=batch, max_seq=src_len)
    dec = dict(family=GPT2, n_layers=6, d_model=768, n_heads=12, head_dim=64, d_ffn=3072, vocab=50265,
               max_pos=1024, dtype="bf16", max_batch=batch, max_seq=tgt_len, max_src=src_len)
    enc.update(kw)
    dec.update(kw)
    return ModelConfig(**enc), ModelConfig(**dec)


def bert_base_config(**kw) -> ModelConfig:
    """BERT-base shape: 12 layers, D=768, 12 heads, GELU FFN 3072, 2 classes, bf16."""
    base = dict(family=BERT, n_layers=12, d_model=768, n_heads=12, head_dim=64, d_ffn=3072,
                vocab=30522, max_pos=512, n_classes=2, dtype="bf16", norm_eps=1e-12,
                max_batch=64, max_seq=128)
    base.update(kw)
    return ModelConfig(**base)


# ----------------------------------------------------------------------------
# weights
# ----------------------------------------------------------------------------

def weight_shapes(cfg: ModelConfig) -> Dict[str, tuple]:
    """Name -> shape of every tensor the model holds (layer names are 0-based storage slots;
    storage slot l is the paper's layer l+1).  Matrices are [out, in]."""
    D, F, V = cfg.d_model, cfg.d_ffn, cfg.vocab
    dq, dkv = cfg.d_q, cfg.d_kv
    m1, m2 = cfg.hsm_m1, cfg.hsm_m2
    s: Dict[str, tuple] = {"tok_emb": (V, D)}
    if cfg.family in (GPT2, BERT):
        s["pos_emb"] = (cfg.max_pos, D)
    if cfg.family == BERT:
        s["type_emb"] = (D,)
        s["emb_ln.g"] = (D,)
        s["emb_ln.b"] = (D,)
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        s[p + "attn_norm.g"] = (D,)
        if cfg.family != LLAMA:
            s[p + "attn_norm.b"] = (D,)
        s[p + "wq"] = (dq, D)
        s[p + "wk"] = (dkv, D)
        s[p + "wv"] = (dkv, D)
        s[p + "wo"] = (D, dq)
        if cfg.family != LLAMA:
            for b, n in (("bq", dq), ("bk", dkv), ("bv", dkv), ("bo", D)):
                s[p + b] = (n,)
        s[p + "ffn_norm.g"] = (D,)
        if cfg.family != LLAMA:
            s[p + "ffn_norm.b"] = (D,)
        if cfg.max_src > 0:   # cross-attention sublayer (encoder-decoder decoders)
            s[p + "cross_norm.g"] = (D,)
            s[p + "cross_norm.b"] = (D,)
            s[p + "cwq"] = (dq, D)
            s[p + "cwk"] = (dkv, D)
            s[p + "cwv"] = (dkv, D)
            s[p + "cwo"] = (D, dq)
            for b, n in (("cbq", dq), ("cbk", dkv), ("cbv", dkv), ("cbo", D)):
                s[p + b] = (n,)
        if cfg.family == LLAMA:
            s[p + "w_gate"] = (F, D)
            s[p + "w_up"] = (F, D)
            s[p + "w_down"] = (D, F)
        else:
            s[p + "w_fc"] = (F, D)
            s[p + "b_fc"] = (F,)
            s[p + "w_proj"] = (D, F)
            s[p + "b_proj"] = (D,)
    if cfg.family == LLAMA:
        s["final_norm.g"] = (D,)
        s["lm_head"] = (V, D)
    elif cfg.family == GPT2:
        s["final_norm.g"] = (D,)
        s["final_norm.b"] = (D,)
    else:
        s["pool.w"] = (D, D)
        s["pool.b"] = (D,)
        s["cls.w"] = (cfg.n_classes, D)
        s["cls.b"] = (cfg.n_classes,)
    s.update({
        "hsm.g0": (D,), "hsm.conv_w": (3, 3), "hsm.conv_b": (1,),
        "hsm.fc1_w": (m1, D), "hsm.fc1_b": (m1,),
        "hsm.fc2_w": (m2, m1), "hsm.fc2_b": (m2,),
        "hsm.fc3_w": (m1, m2), "hsm.fc3_b": (m1,),
        "hsm.g1": (m1,),
        "hsm.fc4_w": (D, m1), "hsm.fc4_b": (D,),
        "hsm.g2": (D,),
    })
    return s


def _is_gain(name: str) -> bool:
    return name.endswith(".g") or name in ("hsm.g0", "hsm.g1", "hsm.g2")


def _is_norm_bias(name: str) -> bool:
    return name.endswith("norm.b") or name.endswith("ln.b")


def make_weight(cfg: ModelConfig, name: str, shape, seed: int = 0, std: float = 0.02,
                gain_std: Optional[float] = None, device="cpu") -> torch.Tensor:
    """One tensor of the synthetic model.

    Matrices, biases and embeddings are N(0, std^2).  Norm gains are 1 + N(0, gain_std^2)
    and norm biases N(0, gain_std^2) with gain_std defaulting to 0 for bf16 models (the
    usual ones/zeros init of a freshly initialised model) and 0.1 for fp32 models, so the
    fp32 parity configurations exercise every gain and bias.  The 3x3 HSM convolution
    gets std 0.5 so that its output is on the scale of its normalised inputs.
    """
    if gain_std is None:
        gain_std = 0.0 if cfg.dtype == "bf16" else 0.1
    dt = cfg.torch_dtype
    if _is_gain(name):
        if gain_std == 0.0:
            return torch.ones(shape, dtype=dt, device=device)
        return normal(seed, name, shape, std=gain_std, mean=1.0, dtype=dt, device=device)
    if _is_norm_bias(name):
        if gain_std == 0.0:
            return torch.zeros(shape, dtype=dt, device=device)
        return normal(seed, name, shape, std=gain_std, dtype=dt, device=device)
    if name == "hsm.conv_w":
        return normal(seed, name, shape, std=0.5, dtype=dt, device=device)
    return normal(seed, name, shape, std=std, dtype=dt, device=device)


def make_weights(cfg: ModelConfig, seed: int = 0, std: float = 0.02,
                 gain_std: Optional[float] = None, device="cpu",
                 overrides: Optional[Dict[str, torch.Tensor]] = None) -> Dict[str, torch.Tensor]:
    out = {}
    for name, shape in weight_shapes(cfg).items():
        if overrides and name in overrides:
            out[name] = overrides[name].to(device=device, dtype=cfg.torch_dtype).reshape(shape)
        else:
            out[name] = make_weight(cfg, name, shape, seed, std, gain_std, device)
    return out


# ----------------------------------------------------------------------------
# prompts, forced-exit laws, KV-fill microbenchmark inputs
# ----------------------------------------------------------------------------

def make_tokens(seed: int, batch: int, length: int, vocab: int, name: str = "tokens") -> torch.Tensor:
    return randint(seed, name, batch * length, 0, vocab - 1).view(batch, length)


def forced_exits_uniform(seed: int, n: int, lo: int, hi: int, name: str = "forced") -> torch.Tensor:
    """Per-token exit layer, integer-uniform on [lo, hi] (1-based layers)."""
    return randint(seed, name, n, lo, hi)


def forced_exits_truncnorm(seed: int, n: int, mean: float, sd: float, lo: int, hi: int,
                           name: str = "forced") -> torch.Tensor:
    """Per-token exit layer from N(mean, sd^2) truncated to [lo, hi], rounded to nearest.

    Drawn by inverting the normal CDF on the truncated range (one uniform per token).
    """
    u = uniform(seed, name, n)
    a = torch.special.ndtr(torch.tensor((lo - mean) / sd, dtype=torch.float64))
    b = torch.special.ndtr(torch.tensor((hi - mean) / sd, dtype=torch.float64))
    z = torch.special.ndtri(a + u * (b - a))
    x = torch.round(mean + sd * z).clamp(lo, hi)
    return x.to(torch.int32)


def make_mapped_states(seed: int, n: int, d: int, dtype=torch.bfloat16, device="cpu",
                       name: str = "mapped") -> torch.Tensor:
    """Exit-state rows s~ ~ N(0, 1) for the skipped-layer KV-fill microbenchmark."""
    return normal(seed, name, (n, d), std=1.0, dtype=dtype, device=device)


# ----------------------------------------------------------------------------
# HSM training batches
# ----------------------------------------------------------------------------

def hsm_train_batch(cfg: ModelConfig, n: int, seed: int = 0, std: float = 1.0):
    """n synthetic training examples of the Hidden State Mapper: (s_i, s_{i-1}, I, target).

    Recipe: s_{i-1} ~ N(0, std^2) per element; s_i = s_{i-1} + N(0, (0.3 std)^2) (a layer's
    residual update); I = (k - 1) unit(s_{i-1}) + N(0, 0.1^2) with the exit layer k uniform on
    [2, N - 1] (the inertia sums k - 1 unit vectors of similar direction); the target is a
    uniform token id on [0, vocab).  Returned as float32 [n, D] tensors and int32 [n]."""
    D = cfg.d_model
    s_prev = normal(seed, "hsm-train-s-prev", (n, D), std=std)
    s_i = s_prev + normal(seed, "hsm-train-delta", (n, D), std=0.3 * std)
    k = randint(seed, "hsm-train-layer", n, 2, max(2, cfg.n_layers - 1)).to(torch.float32)
    u = s_prev / s_prev.norm(dim=1, keepdim=True).clamp_min(1e-30)
    inertia = (k - 1)[:, None] * u + normal(seed, "hsm-train-inertia", (n, D), std=0.1)
    target = randint(seed, "hsm-train-target", n, 0, cfg.vocab - 1)
    return s_i.contiguous(), s_prev.contiguous(), inertia.contiguous(), target


def hsm_cls_batch(cfg: ModelConfig, n: int, n_cls: int, seed: int = 0, std: float = 1.0):
    """n synthetic encoder training examples of the Hidden State Mapper for classification:
    (s_i, s_{i-1}, I, s_N, labels).

    Recipe: s_i, s_{i-1} and I as in hsm_train_batch; the original final state s_N =
    s_i + N(0, (0.5 std)^2) (the remaining layers' residual updates); the first n_cls rows are
    the labelled [CLS] rows, labels uniform on [0, n_classes).  Returned as float32 [n, D]
    tensors and int32 [n_cls]."""
    s_i, s_prev, inertia, _ = hsm_train_batch(cfg, n, seed=seed, std=std)
    s_final = s_i + normal(seed, "hsm-cls-final", (n, cfg.d_model), std=0.5 * std)
    labels = randint(seed, "hsm-cls-label", n_cls, 0, max(0, cfg.n_classes - 1))
    return s_i, s_prev, inertia, s_final.contiguous(), labels
