"""Plain CPU oracle of one HSM training step (float64, PyTorch CPU autograd).

TEST INFRASTRUCTURE ONLY: imported by the test suite alone; the library never imports it
and shares no code with it.

What it follows: the Hidden State Mapper is trained with the base model frozen (Sec. 4.2;
Sec. 5.1 "Training"): its mapped state s~ goes through the frozen final norm and LM head
("linearly transformed into token-level distributions"), and the cross-entropy against
the next input token (labels = one-position-shifted input tokens) is minimised with AdamW
(App. D: learning rates 1e-3 .. 1e-5, weight decay 0 .. 1e-2).

* The HSM forward is Table S1 (App. B) as in ``adept_oracle.OracleModel.hsm``, written with
  torch ops so that autograd gives the gradients: three separately RMS-normalised rows (shared
  gain g0), a 3x3 convolution with padding (0, 1), FC1 and FC2 with erf-GELU, FC3, RMSNorm
  with gain g1 plus FC1's output, FC4, RMSNorm with gain g2 plus the convolution output.
* The loss is the mean over the n examples of -log softmax(logits)[target].
* Classification (encoders, Sec. 4.3): with no next token to predict, the mapped state is
  pulled toward the original final hidden state s_N of the same token by a similarity loss,
  and the task loss of the frozen pooler and classifier is added.  Read here as: similarity
  loss = mean over the n examples of 1 - cos(s~, s_N) (cos taken as 0 where a norm is 0);
  task loss = softmax cross-entropy of the classifier's logits on the pooled mapped state of
  the first n_cls examples (the [CLS] rows that carry a label; with two classes this is the
  binary cross-entropy of the class-1 probability), averaged over those rows and weighted by
  cls_weight (1 by default: the paper adds the two).
* AdamW is the decoupled-weight-decay Adam of Loshchilov & Hutter, written out: m = b1 m +
  (1 - b1) g, v = b2 v + (1 - b2) g^2, theta -= lr (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) +
  eps) + lr wd theta (the decay applied to the parameter before this step's update).
* Precision: float64 throughout.  With ``bf16=True`` every linear layer (the four FCs, the
  LM head, the pooler and the classifier) rounds its inputs to bfloat16 the way the library's bf16 models feed their tensor cores:
  the forward product takes round(x) and round(W); the input gradient takes round(g) and
  round(W); the weight gradient takes round(g) and round(x).  Bias gradients, norms,
  activations, the loss and the optimiser stay unrounded.  (The paper fixes no training
  precision; this is the same GEMM-input rounding the inference oracle applies.)
"""
from __future__ import annotations

from typing import Dict, List, Optional, Tuple

import numpy as np
import torch
import torch.nn.functional as F

LLAMA, GPT2, BERT = 0, 1, 2

HSM_PARAMS: List[str] = ["hsm.g0", "hsm.conv_w", "hsm.conv_b", "hsm.fc1_w", "hsm.fc1_b", "hsm.fc2_w", "hsm.fc2_b",
                         "hsm.fc3_w", "hsm.fc3_b", "hsm.g1", "hsm.fc4_w", "hsm.fc4_b", "hsm.g2"]


def _t(x) -> torch.Tensor:
    return (x if torch.is_tensor(x) else torch.as_tensor(np.asarray(x))).double()


def rmsnorm(x: torch.Tensor, g: torch.Tensor, eps: float) -> torch.Tensor:
    return x * torch.rsqrt(torch.mean(x * x, dim=-1, keepdim=True) + eps) * g


def round_bf16(x: torch.Tensor) -> torch.Tensor:
    """Nearest bfloat16 (ties to even) of the float32 value, as float64."""
    return x.to(torch.float32).to(torch.bfloat16).to(torch.float64)


class _Linear(torch.autograd.Function):
    """y = x W^T + b whose three products take (optionally bf16-rounded) inputs."""

    @staticmethod
    def forward(ctx, x, W, b, rnd: bool):
        R = round_bf16 if rnd else (lambda t: t)
        xr, Wr = R(x), R(W)
        ctx.save_for_backward(xr, Wr)
        ctx.rnd = rnd
        y = xr @ Wr.T
        return y if b is None else y + b

    @staticmethod
    def backward(ctx, g):
        xr, Wr = ctx.saved_tensors
        gr = round_bf16(g) if ctx.rnd else g
        gx = gr @ Wr
        gW = gr.T @ xr
        return gx, gW, (g.sum(0) if ctx.needs_input_grad[2] else None), None


def linear(x, W, b, rnd: bool):
    return _Linear.apply(x, W, b, rnd)


def hsm_forward(p: Dict[str, torch.Tensor], cfg, s_i, s_prev, inertia, bf16: bool = False) -> torch.Tensor:
    """Table S1 (App. B) on rows [n, D]; p holds the HSM parameters (float64 tensors)."""
    eps = cfg.hsm_eps
    X = torch.stack([rmsnorm(_t(s_i), p["hsm.g0"], eps), rmsnorm(_t(s_prev), p["hsm.g0"], eps),
                     rmsnorm(_t(inertia), p["hsm.g0"], eps)], dim=1)            # [n, 3, D]
    c0 = F.conv2d(X[:, None], p["hsm.conv_w"][None, None], p["hsm.conv_b"], padding=(0, 1))[:, 0, 0]   # [n, D]
    h1 = F.gelu(linear(c0, p["hsm.fc1_w"], p["hsm.fc1_b"], bf16))
    h2 = F.gelu(linear(h1, p["hsm.fc2_w"], p["hsm.fc2_b"], bf16))
    h3 = linear(h2, p["hsm.fc3_w"], p["hsm.fc3_b"], bf16)
    h4 = rmsnorm(h3, p["hsm.g1"], eps) + h1
    h5 = linear(h4, p["hsm.fc4_w"], p["hsm.fc4_b"], bf16)
    return rmsnorm(h5, p["hsm.g2"], eps) + c0


def head_logits(W: Dict[str, object], cfg, x: torch.Tensor, bf16: bool = False) -> torch.Tensor:
    """The frozen final norm and LM head of a decoder."""
    if cfg.family == LLAMA:
        return linear(rmsnorm(x, _t(W["final_norm.g"]), cfg.norm_eps), _t(W["lm_head"]), None, bf16)
    y = F.layer_norm(x, (cfg.d_model,), _t(W["final_norm.g"]), _t(W["final_norm.b"]), cfg.norm_eps)
    return linear(y, _t(W["tok_emb"]), None, bf16)


def hsm_loss(p: Dict[str, torch.Tensor], W, cfg, s_i, s_prev, inertia, targets, bf16: bool = False) -> torch.Tensor:
    """Mean cross-entropy of the head's distribution of the mapped state against the targets."""
    logits = head_logits(W, cfg, hsm_forward(p, cfg, s_i, s_prev, inertia, bf16), bf16)
    return F.cross_entropy(logits, torch.as_tensor(np.asarray(targets), dtype=torch.long))


def cls_head_logits(W: Dict[str, object], cfg, x: torch.Tensor, bf16: bool = False) -> torch.Tensor:
    """The frozen pooler (dense + tanh) and classifier of an encoder, applied to final states."""
    pooled = torch.tanh(linear(x, _t(W["pool.w"]), _t(W["pool.b"]), bf16))
    return linear(pooled, _t(W["cls.w"]), _t(W["cls.b"]), bf16)


def cosine_rows(a: torch.Tensor, b: torch.Tensor) -> torch.Tensor:
    """cos of each row pair, a.b / (|a| |b|), and 0 where |a| |b| = 0."""
    den = torch.sqrt(torch.clamp_min((a * a).sum(-1) * (b * b).sum(-1), 1e-300))
    return (a * b).sum(-1) / den


def hsm_cls_loss(p: Dict[str, torch.Tensor], W, cfg, s_i, s_prev, inertia, s_final, labels, cls_weight: float = 1.0,
                 bf16: bool = False) -> torch.Tensor:
    """Similarity loss against the original final states plus the weighted task loss of the
    first len(labels) rows (Sec. 4.3)."""
    st = hsm_forward(p, cfg, s_i, s_prev, inertia, bf16)
    loss = torch.mean(1.0 - cosine_rows(st, _t(s_final)))
    lab = torch.as_tensor(np.asarray(labels), dtype=torch.long).reshape(-1)
    if lab.numel():
        loss = loss + cls_weight * F.cross_entropy(cls_head_logits(W, cfg, st[:lab.numel()], bf16), lab)
    return loss


def adamw_update(theta: np.ndarray, g: np.ndarray, m: np.ndarray, v: np.ndarray, t: int, lr: float, b1: float,
                 b2: float, eps: float, wd: float) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """One AdamW step (decoupled weight decay, bias-corrected moments) of one parameter."""
    m = b1 * m + (1.0 - b1) * g
    v = b2 * v + (1.0 - b2) * g * g
    mhat = m / (1.0 - b1 ** t)
    vhat = v / (1.0 - b2 ** t)
    theta = theta - lr * wd * theta - lr * mhat / (np.sqrt(vhat) + eps)
    return theta, m, v


def hsm_train_step(W: Dict[str, object], cfg, s_i, s_prev, inertia, targets, lr: float, b1: float, b2: float,
                   eps: float, wd: float, t: int, params: Optional[Dict[str, np.ndarray]] = None,
                   state: Optional[Dict[str, Tuple[np.ndarray, np.ndarray]]] = None, bf16: bool = False):
    """Loss (before the update), the gradients, the updated parameters and AdamW state.

    params / state: the HSM parameters and (m, v) moments of the previous step (default:
    the model's HSM weights, zero moments); t: this step's number (1 for the first)."""
    return _step(lambda p: hsm_loss(p, W, cfg, s_i, s_prev, inertia, targets, bf16), W, lr, b1, b2, eps, wd, t,
                 params, state)


def hsm_cls_train_step(W: Dict[str, object], cfg, s_i, s_prev, inertia, s_final, labels, cls_weight: float, lr: float,
                       b1: float, b2: float, eps: float, wd: float, t: int,
                       params: Optional[Dict[str, np.ndarray]] = None,
                       state: Optional[Dict[str, Tuple[np.ndarray, np.ndarray]]] = None, bf16: bool = False):
    """The encoder (classification) training step of Sec. 4.3: as hsm_train_step with
    hsm_cls_loss; labels belong to the first len(labels) examples."""
    return _step(lambda p: hsm_cls_loss(p, W, cfg, s_i, s_prev, inertia, s_final, labels, cls_weight, bf16), W, lr, b1,
                 b2, eps, wd, t, params, state)


def _step(loss_fn, W, lr, b1, b2, eps, wd, t, params, state):
    if params is None:
        params = {k: np.asarray(_t(W[k])) for k in HSM_PARAMS}
    if state is None:
        state = {k: (np.zeros_like(params[k]), np.zeros_like(params[k])) for k in HSM_PARAMS}
    p = {k: torch.tensor(params[k], dtype=torch.float64, requires_grad=True) for k in HSM_PARAMS}
    loss = loss_fn(p)
    loss.backward()
    grads = {k: p[k].grad.numpy().copy() for k in HSM_PARAMS}
    new_params, new_state = {}, {}
    for k in HSM_PARAMS:
        th, m, v = adamw_update(params[k], grads[k], state[k][0], state[k][1], t, lr, b1, b2, eps, wd)
        new_params[k], new_state[k] = th, (m, v)
    return float(loss.item()), grads, new_params, new_state
