"""Python binding of libadept.so (include/adept.h): argument marshalling only.

Every step of the early-exit pass runs in the library's CUDA kernels; this module
passes torch device pointers and the CUDA stream through ctypes and turns a non-OK
status into an exception.  There is no fallback: if the library is not built, every
call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libadept.so")

ADEPT_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "OOM", 3: "CAPACITY", 4: "CUDA", 5: "TIMEOUT", 6: "DEVICE_INPUT"}
FAMILY = {"llama": 0, "gpt2": 1, "bert": 2}
OPT_HSM_IDENTITY, OPT_PROFILE, OPT_GEMM_SIMT, OPT_DECODE_GRAPH, OPT_DECODE_GEMM = 1, 2, 3, 4, 5
OPT_EXIT_METRIC, OPT_ALL_AT_ONCE, OPT_STOP_ENTIRELY, OPT_DECODE_STREAM, OPT_DECODE_TILED = 7, 8, 9, 10, 11
OPT_SPAN_TIMER, OPT_ATTN_TC, OPT_FUSED_EXIT = 12, 13, 14
EXIT_GLOBAL, EXIT_LOCAL, EXIT_BOTH = 0, 1, 2
PROF_GEMM_PREFILL, PROF_KV_FILL, PROF_ATTENTION, PROF_GEMM_DECODE, PROF_GEMM_TRAIN = 0, 1, 2, 3, 4
HSM_PARAMS, HSM_GRADS, HSM_MOMENT1, HSM_MOMENT2 = 0, 1, 2, 3
# HSM parameters in the order of adept_hsm_train_read's `param` (Table S1)
HSM_PARAM_NAMES = ["hsm.g0", "hsm.conv_w", "hsm.conv_b", "hsm.fc1_w", "hsm.fc1_b", "hsm.fc2_w", "hsm.fc2_b",
                   "hsm.fc3_w", "hsm.fc3_b", "hsm.g1", "hsm.fc4_w", "hsm.fc4_b", "hsm.g2"]

# every symbol declared in include/adept.h
ABI_SYMBOLS = [
    "adept_model_load", "adept_prefill", "adept_decode_step", "adept_skip_kv_fill", "adept_free",
    "adept_last_error", "adept_status_string", "adept_seq_reserve", "adept_read_kv",
    "adept_read_final_states", "adept_check_device_status", "adept_set_option", "adept_profile_read",
    "adept_launch_count", "adept_skip_kv_fill_noalloc",
    "adept_calibrate_threshold", "adept_hsm_train_init", "adept_hsm_train_step", "adept_hsm_train_read",
    "adept_hsm_param_numel", "adept_hsm_train_step_cls", "adept_set_wait_limit", "adept_set_alloc_fail_after",
    "adept_span_read", "adept_set_cross_source",
]


class AdeptError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"adept status {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class AdeptConfig(ctypes.Structure):
    _fields_ = [
        ("family", ctypes.c_int), ("n_layers", ctypes.c_int), ("d_model", ctypes.c_int),
        ("n_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
        ("d_ffn", ctypes.c_int), ("vocab", ctypes.c_int), ("max_pos", ctypes.c_int),
        ("n_classes", ctypes.c_int), ("dtype", ctypes.c_int), ("norm_eps", ctypes.c_float),
        ("rope_theta", ctypes.c_float), ("hsm_eps", ctypes.c_float), ("hsm_m1", ctypes.c_int),
        ("hsm_m2", ctypes.c_int), ("kv_block_tokens", ctypes.c_int), ("max_batch", ctypes.c_int),
        ("max_seq", ctypes.c_int), ("kv_pool_blocks", ctypes.c_int), ("max_pass_tokens", ctypes.c_int),
        ("block_shuffle_seed", ctypes.c_uint64), ("max_src", ctypes.c_int),
    ]


class AdeptTensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("data", ctypes.c_void_p), ("numel", ctypes.c_int64)]


class AdeptAdamW(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float)]


class AdeptTensorTable(ctypes.Structure):
    _fields_ = [("tensors", ctypes.POINTER(AdeptTensor)), ("n_tensors", ctypes.c_int)]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load libadept.so (raises if it is missing: there is no CPU fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is not built; call paper_2601_03700_gb300.build.build() first")
    lib = ctypes.CDLL(path)
    vp, i32p, fp, st = ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p
    c_int, c_float = ctypes.c_int, ctypes.c_float
    lib.adept_model_load.argtypes = [ctypes.POINTER(AdeptConfig), ctypes.POINTER(AdeptTensorTable), st,
                                     ctypes.POINTER(ctypes.c_void_p)]
    lib.adept_prefill.argtypes = [vp, c_int, c_int, i32p, c_float, i32p, i32p, fp, i32p, fp, st]
    lib.adept_decode_step.argtypes = [vp, c_int, i32p, c_float, i32p, i32p, fp, i32p, fp, st]
    lib.adept_skip_kv_fill.argtypes = [vp, c_int, vp, i32p, i32p, i32p, st]
    lib.adept_skip_kv_fill_noalloc.argtypes = [vp, c_int, vp, i32p, i32p, i32p, st]
    lib.adept_free.argtypes = [vp]
    lib.adept_free.restype = None
    lib.adept_last_error.argtypes = [vp]
    lib.adept_last_error.restype = ctypes.c_char_p
    lib.adept_status_string.argtypes = [c_int]
    lib.adept_status_string.restype = ctypes.c_char_p
    lib.adept_seq_reserve.argtypes = [vp, c_int, ctypes.POINTER(ctypes.c_int32)]
    lib.adept_read_kv.argtypes = [vp, c_int, c_int, c_int, c_int, vp, vp, st]
    lib.adept_read_final_states.argtypes = [vp, fp, c_int, st]
    lib.adept_check_device_status.argtypes = [vp, st]
    lib.adept_set_option.argtypes = [vp, c_int, c_int]
    lib.adept_profile_read.argtypes = [vp, c_int, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_double),
                                       ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
    lib.adept_set_cross_source.argtypes = [vp, c_int, ctypes.POINTER(ctypes.c_int32), fp, st]
    lib.adept_set_cross_source.restype = c_int
    lib.adept_span_read.argtypes = [vp, c_int, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_double)]
    lib.adept_span_read.restype = c_int
    lib.adept_launch_count.argtypes = [vp]
    lib.adept_launch_count.restype = ctypes.c_int64
    lib.adept_calibrate_threshold.argtypes = [vp, c_int, c_int, i32p, c_float, c_float, c_int, c_float, c_float,
                                              ctypes.POINTER(c_float), ctypes.POINTER(c_float),
                                              ctypes.POINTER(c_int), st]
    lib.adept_calibrate_threshold.restype = c_int
    lib.adept_hsm_train_init.argtypes = [vp, c_int, st]
    lib.adept_hsm_train_init.restype = c_int
    lib.adept_hsm_train_step.argtypes = [vp, c_int, fp, fp, fp, i32p, ctypes.POINTER(AdeptAdamW), fp, st]
    lib.adept_hsm_train_step.restype = c_int
    lib.adept_hsm_train_step_cls.argtypes = [vp, c_int, fp, fp, fp, fp, c_int, i32p, ctypes.c_float,
                                             ctypes.POINTER(AdeptAdamW), fp, st]
    lib.adept_hsm_train_step_cls.restype = c_int
    lib.adept_hsm_train_read.argtypes = [vp, c_int, c_int, fp, ctypes.c_int64, st]
    lib.adept_hsm_train_read.restype = c_int
    lib.adept_set_wait_limit.argtypes = [ctypes.c_int64]
    lib.adept_set_wait_limit.restype = c_int
    lib.adept_set_alloc_fail_after.argtypes = [ctypes.c_int64]
    lib.adept_set_alloc_fail_after.restype = None
    lib.adept_hsm_param_numel.argtypes = [vp, c_int]
    lib.adept_hsm_param_numel.restype = ctypes.c_int64
    for name in ABI_SYMBOLS:
        fn = getattr(lib, name)
        if fn.restype is ctypes.c_int or name in ("adept_model_load", "adept_prefill", "adept_decode_step",
                                                   "adept_skip_kv_fill", "adept_skip_kv_fill_noalloc",
                                                   "adept_seq_reserve", "adept_read_kv",
                                                   "adept_read_final_states", "adept_check_device_status",
                                                   "adept_set_option", "adept_profile_read"):
            fn.restype = c_int
    _lib = lib
    return lib


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to the library must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        if not torch.cuda.is_available():
            return ctypes.c_void_p(None)
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(lib, model_handle, status: int):
    if status != ADEPT_OK:
        msg = lib.adept_last_error(model_handle).decode(errors="replace")
        raise AdeptError(status, msg)


def make_config(cfg) -> AdeptConfig:
    """adept_config from any object with the fields of include/adept.h (e.g. synth.ModelConfig)."""
    g = lambda k, d=0: getattr(cfg, k, d)  # noqa: E731
    dt = g("dtype", "bf16")
    dt = {"f32": 0, "fp32": 0, "float32": 0, "bf16": 1, "bfloat16": 1}.get(dt, dt)
    fam = g("family", 0)
    fam = FAMILY.get(fam, fam)
    return AdeptConfig(
        family=int(fam), n_layers=g("n_layers"), d_model=g("d_model"), n_heads=g("n_heads"),
        n_kv_heads=g("n_kv_heads", 0) or 0, head_dim=g("head_dim"), d_ffn=g("d_ffn"), vocab=g("vocab"),
        max_pos=g("max_pos", 0) or 0, n_classes=g("n_classes", 0) or 0, dtype=int(dt),
        norm_eps=float(g("norm_eps", 1e-5)), rope_theta=float(g("rope_theta", 10000.0)),
        hsm_eps=float(g("hsm_eps", 1e-6)), hsm_m1=g("hsm_m1"), hsm_m2=g("hsm_m2"),
        kv_block_tokens=g("kv_block_tokens", 16), max_batch=g("max_batch"), max_seq=g("max_seq"),
        kv_pool_blocks=g("kv_pool_blocks", 0) or 0, max_pass_tokens=g("max_pass_tokens", 0) or 0,
        block_shuffle_seed=int(g("block_shuffle_seed", 0) or 0), max_src=int(g("max_src", 0) or 0))


# ---------------------------------------------------------------------------
# functions with the ABI's names
# ---------------------------------------------------------------------------

def adept_model_load(cfg, weights: Dict[str, torch.Tensor], stream=None):
    """Returns an opaque model handle.  Weight tensors may live on the host or the device."""
    lib = load_library()
    c = make_config(cfg)
    names = list(weights.keys())
    keep = [weights[n].contiguous() for n in names]
    arr = (AdeptTensor * len(names))()
    enc = [n.encode() for n in names]
    for i, (n, t) in enumerate(zip(enc, keep)):
        arr[i] = AdeptTensor(n, t.data_ptr(), t.numel())
    table = AdeptTensorTable(arr, len(names))
    h = ctypes.c_void_p()
    st = lib.adept_model_load(ctypes.byref(c), ctypes.byref(table), _stream(stream), ctypes.byref(h))
    _check(lib, None, st)
    return h


def adept_prefill(m, batch: int, prompt_len: int, tokens: torch.Tensor, delta: float,
                  forced: Optional[torch.Tensor] = None, exit_layer_out: Optional[torch.Tensor] = None,
                  logits_out: Optional[torch.Tensor] = None, next_token_out: Optional[torch.Tensor] = None,
                  sim_out: Optional[torch.Tensor] = None, stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_prefill(m, batch, prompt_len, _ptr(tokens), float(delta), _ptr(forced),
                                      _ptr(exit_layer_out), _ptr(logits_out), _ptr(next_token_out), _ptr(sim_out),
                                      _stream(stream)))


def adept_decode_step(m, batch: int, tokens: torch.Tensor, delta: float, forced: Optional[torch.Tensor] = None,
                      exit_layer_out: Optional[torch.Tensor] = None, logits_out: Optional[torch.Tensor] = None,
                      next_token_out: Optional[torch.Tensor] = None, sim_out: Optional[torch.Tensor] = None,
                      stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_decode_step(m, batch, _ptr(tokens), float(delta), _ptr(forced), _ptr(exit_layer_out),
                                          _ptr(logits_out), _ptr(next_token_out), _ptr(sim_out), _stream(stream)))


def adept_skip_kv_fill(m, n_tokens: int, h_mapped: torch.Tensor, exit_layer: torch.Tensor, seq: torch.Tensor,
                       pos: torch.Tensor, stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_skip_kv_fill(m, n_tokens, _ptr(h_mapped), _ptr(exit_layer), _ptr(seq), _ptr(pos),
                                           _stream(stream)))


def adept_skip_kv_fill_noalloc(m, n_tokens: int, h_mapped: torch.Tensor, exit_layer: torch.Tensor,
                               seq: torch.Tensor, pos: torch.Tensor, stream=None):
    """adept_skip_kv_fill with its scratch in a fixed device array (no allocation)."""
    lib = load_library()
    _check(lib, m, lib.adept_skip_kv_fill_noalloc(m, n_tokens, _ptr(h_mapped), _ptr(exit_layer), _ptr(seq),
                                                   _ptr(pos), _stream(stream)))


def adept_calibrate_threshold(m, batch: int, prompt_len: int, tokens: torch.Tensor, target_rdc: float,
                              tol: float = 0.005, max_iter: int = 24, lo: float = -1.0, hi: float = 1.0,
                              stream=None):
    """Bisection on the exit threshold to a target reduction in computation over the
    calibration batch (Sec. 4.1, Sec. 5.1).  Returns (delta, rdc, passes)."""
    lib = load_library()
    d, r, n = ctypes.c_float(), ctypes.c_float(), ctypes.c_int()
    _check(lib, m, lib.adept_calibrate_threshold(m, batch, prompt_len, _ptr(tokens), target_rdc, tol, max_iter, lo, hi,
                                                 ctypes.byref(d), ctypes.byref(r), ctypes.byref(n), _stream(stream)))
    return d.value, r.value, n.value


def adept_hsm_train_init(m, max_rows: int, stream=None):
    """Master parameters from the model's HSM weights, zero AdamW moments, workspaces for
    max_rows examples per step (Sec. 4.2; App. D)."""
    lib = load_library()
    _check(lib, m, lib.adept_hsm_train_init(m, int(max_rows), _stream(stream)))


def adept_hsm_train_step(m, n: int, s_i: torch.Tensor, s_prev: torch.Tensor, inertia: torch.Tensor,
                         target: torch.Tensor, lr: float, beta1: float = 0.9, beta2: float = 0.999,
                         eps: float = 1e-8, weight_decay: float = 0.0, loss_out: Optional[torch.Tensor] = None,
                         stream=None):
    """One HSM training step: cross-entropy of the mapped state through the frozen head
    against the target tokens, backward, AdamW."""
    lib = load_library()
    hp = AdeptAdamW(lr, beta1, beta2, eps, weight_decay)
    _check(lib, m, lib.adept_hsm_train_step(m, int(n), _ptr(s_i), _ptr(s_prev), _ptr(inertia), _ptr(target),
                                             ctypes.byref(hp), _ptr(loss_out), _stream(stream)))


def adept_hsm_train_step_cls(m, n: int, s_i: torch.Tensor, s_prev: torch.Tensor, inertia: torch.Tensor,
                             s_final: torch.Tensor, labels: Optional[torch.Tensor], lr: float, cls_weight: float = 1.0,
                             beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.0,
                             loss_out: Optional[torch.Tensor] = None, stream=None):
    """One encoder HSM training step (Sec. 4.3): similarity loss against the original final
    states plus cls_weight times the classifier's cross-entropy on the first len(labels)
    rows, backward, AdamW."""
    lib = load_library()
    hp = AdeptAdamW(lr, beta1, beta2, eps, weight_decay)
    n_cls = 0 if labels is None else labels.numel()
    _check(lib, m, lib.adept_hsm_train_step_cls(m, int(n), _ptr(s_i), _ptr(s_prev), _ptr(inertia), _ptr(s_final),
                                                 int(n_cls), _ptr(labels), float(cls_weight), ctypes.byref(hp),
                                                 _ptr(loss_out), _stream(stream)))


def adept_hsm_train_read(m, what: int, param: int, out: torch.Tensor, stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_hsm_train_read(m, int(what), int(param), _ptr(out), out.numel(), _stream(stream)))


def adept_hsm_param_numel(m, param: int) -> int:
    return int(load_library().adept_hsm_param_numel(m, int(param)))


def adept_free(m):
    if m:
        load_library().adept_free(m)


def adept_seq_reserve(m, lens):
    lib = load_library()
    arr = (ctypes.c_int32 * len(lens))(*[int(x) for x in lens])
    _check(lib, m, lib.adept_seq_reserve(m, len(lens), arr))


def adept_read_kv(m, layer: int, seq: int, pos0: int, n_pos: int, k_out: torch.Tensor, v_out: torch.Tensor,
                  stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_read_kv(m, layer, seq, pos0, n_pos, _ptr(k_out), _ptr(v_out), _stream(stream)))


def adept_read_final_states(m, out: torch.Tensor, rows: int, stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_read_final_states(m, _ptr(out), rows, _stream(stream)))


def adept_set_cross_source(m, src_len, states: torch.Tensor, stream=None):
    """Cross-attention source of sequences 0..len(src_len)-1: states fp32 [sum(src_len), D] on
    the device, in sequence order."""
    lib = load_library()
    n = len(src_len)
    arr = (ctypes.c_int32 * n)(*[int(x) for x in src_len])
    _check(lib, m, lib.adept_set_cross_source(m, n, arr, _ptr(states), _stream(stream)))


def adept_check_device_status(m, stream=None):
    lib = load_library()
    _check(lib, m, lib.adept_check_device_status(m, _stream(stream)))


def adept_set_option(m, option: int, value: int):
    lib = load_library()
    _check(lib, m, lib.adept_set_option(m, option, value))


def adept_profile_read(m, cls: int):
    lib = load_library()
    n = ctypes.c_int64()
    ms, fl, by = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(lib, m, lib.adept_profile_read(m, cls, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(fl),
                                           ctypes.byref(by)))
    return n.value, ms.value, fl.value, by.value


def adept_span_read(m, cls: int):
    """(launches, summed in-situ spans in ms) of class `cls` recorded by the span timer."""
    lib = load_library()
    n = ctypes.c_int64()
    ms = ctypes.c_double()
    _check(lib, m, lib.adept_span_read(m, cls, ctypes.byref(n), ctypes.byref(ms)))
    return n.value, ms.value


def adept_launch_count(m) -> int:
    return int(load_library().adept_launch_count(m))


def adept_set_wait_limit(cycles: int):
    lib = load_library()
    _check(lib, None, lib.adept_set_wait_limit(int(cycles)))


def adept_set_alloc_fail_after(n: int):
    load_library().adept_set_alloc_fail_after(int(n))


# ---------------------------------------------------------------------------
# a small convenience wrapper (allocates outputs with torch, which is plumbing)
# ---------------------------------------------------------------------------

class Model:
    def __init__(self, cfg, weights: Dict[str, torch.Tensor], stream=None):
        self.cfg = cfg
        self.h = adept_model_load(cfg, weights, stream)
        self.n_out = cfg.n_classes if FAMILY.get(getattr(cfg, "family", 0), getattr(cfg, "family", 0)) == 2 \
            else cfg.vocab

    def close(self):
        if self.h:
            adept_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _outs(self, n_tok, batch, dev):
        N = self.cfg.n_layers
        return (torch.empty(n_tok, dtype=torch.int32, device=dev),
                torch.empty(batch, self.n_out, dtype=torch.float32, device=dev),
                torch.empty(batch, dtype=torch.int32, device=dev),
                torch.empty(n_tok, N, dtype=torch.float32, device=dev))

    def prefill(self, tokens: torch.Tensor, delta: float, forced: Optional[torch.Tensor] = None, stream=None):
        B, P = tokens.shape
        ex, lg, nx, sim = self._outs(B * P, B, tokens.device)
        adept_prefill(self.h, B, P, tokens.to(torch.int32).contiguous().view(-1), delta,
                      None if forced is None else forced.to(torch.int32).contiguous().view(-1), ex, lg, nx, sim,
                      stream)
        return ex, lg, nx, sim

    def decode_step(self, tokens: torch.Tensor, delta: float, forced: Optional[torch.Tensor] = None, stream=None):
        B = tokens.numel()
        ex, lg, nx, sim = self._outs(B, B, tokens.device)
        adept_decode_step(self.h, B, tokens.to(torch.int32).contiguous().view(-1), delta,
                          None if forced is None else forced.to(torch.int32).contiguous().view(-1), ex, lg, nx, sim,
                          stream)
        return ex, lg, nx, sim

    def set_cross_source(self, src_len, states: torch.Tensor, stream=None):
        adept_set_cross_source(self.h, src_len, states.float().contiguous(), stream)

    def final_states(self, rows: int) -> torch.Tensor:
        out = torch.empty(rows, self.cfg.d_model, dtype=torch.float32, device="cuda")
        adept_read_final_states(self.h, out, rows)
        return out

    def read_kv(self, layer: int, seq: int, pos0: int, n_pos: int):
        dt = torch.bfloat16 if getattr(self.cfg, "dtype", "bf16") in ("bf16", 1) else torch.float32
        kvh = getattr(self.cfg, "n_kv_heads", 0) or self.cfg.n_heads
        k = torch.empty(n_pos, kvh, self.cfg.head_dim, dtype=dt, device="cuda")
        v = torch.empty_like(k)
        adept_read_kv(self.h, layer, seq, pos0, n_pos, k, v)
        return k, v

    def check(self):
        adept_check_device_status(self.h)

    def hsm_train_read(self, what: int, param: int) -> torch.Tensor:
        out = torch.empty(adept_hsm_param_numel(self.h, param), dtype=torch.float32, device="cuda")
        adept_hsm_train_read(self.h, what, param, out)
        return out
