"""Thin ctypes binding of libtadm (include/tadm.h).

Functions keep the C names and only marshal arguments: every step of the
sampling loop runs in the library's CUDA kernels.  PyTorch provides device
memory and streams.  Loading fails loudly when the library is missing; there
is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libtadm.so")

TADM_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "OOM", 5: "TIMEOUT", 6: "STATE"}

ABI_FUNCTIONS = [
    "tadm_weight_count", "tadm_weight_info", "tadm_create", "tadm_destroy", "tadm_last_error",
    "tadm_status_string", "tadm_workspace_size", "tadm_bind_workspace", "tadm_cache_size", "tadm_reset",
    "tadm_prefill", "tadm_anchor_forward", "tadm_denoise_step", "tadm_commit_block", "tadm_generate",
    "tadm_sync_status", "tadm_get_counters", "tadm_plan", "tadm_layer_cost", "tadm_gemm", "tadm_confidence",
    "tadm_topk_unmask", "tadm_attention", "tadm_probe_enable", "tadm_probe_read", "tadm_head_scratch_size",
    "tadm_head_confidence", "tadm_head_confidence_static", "tadm_probe_breakdown",
    "tadm_remdm_schedule", "tadm_remdm_uniforms", "tadm_remdm_update", "tadm_generate_remdm",
    "tadm_eb_update", "tadm_eb_scratch_bytes", "tadm_generate_entropy_bound",
]


class TadmError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class tadm_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "vocab", "d_model", "n_heads", "n_kv_heads", "head_dim", "ffn", "glu", "n_shared", "n_anchor",
        "n_denoise", "fusion", "fusion_rank", "fusion_heads", "dtype", "tied_lm_head")] + [
        ("norm_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)] + [
        (n, ctypes.c_int32) for n in ("sliding_window", "global_every", "qk_norm", "sandwich_norm")] + [
        ("rope_theta_global", ctypes.c_float), ("qkv_split", ctypes.c_int32)]


class tadm_step_outputs(ctypes.Structure):
    _fields_ = [("logits", ctypes.c_void_p), ("conf", ctypes.c_void_p), ("tok", ctypes.c_void_p),
                ("selected", ctypes.c_void_p), ("fused", ctypes.c_void_p)]


class tadm_counters(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "shared_layers", "anchor_layers", "denoise_layers", "anchor_calls", "denoise_steps", "commit_passes",
        "kernel_launches")]


class tadm_plan_event(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("kind", "block", "n", "k")]


_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libtadm.so (built in-tree by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise FileNotFoundError(f"{path} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    P, I, I64, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t
    cfgp = ctypes.POINTER(tadm_config)
    sig = {
        "tadm_weight_count": (I, [cfgp]),
        "tadm_weight_info": (I, [cfgp, I, ctypes.c_char_p, I, ctypes.POINTER(I64), ctypes.POINTER(I64)]),
        "tadm_create": (I, [cfgp, ctypes.POINTER(P), I, I, I, I, ctypes.POINTER(P)]),
        "tadm_destroy": (None, [P]),
        "tadm_last_error": (ctypes.c_char_p, [P]),
        "tadm_status_string": (ctypes.c_char_p, [I]),
        "tadm_workspace_size": (I, [P, ctypes.POINTER(SZ)]),
        "tadm_bind_workspace": (I, [P, P, SZ]),
        "tadm_cache_size": (I, [P, I, I, ctypes.POINTER(SZ)]),
        "tadm_reset": (I, [P, I]),
        "tadm_prefill": (I, [P, P, I, I, P]),
        "tadm_anchor_forward": (I, [P, P, I, I, I, P, P]),
        "tadm_denoise_step": (I, [P, P, I, I, I, I, I, P, ctypes.POINTER(tadm_step_outputs), P]),
        "tadm_commit_block": (I, [P, P, I, I, P]),
        "tadm_generate": (I, [P, P, I, I, P, I, I, I, I, P]),
        "tadm_sync_status": (I, [P]),
        "tadm_get_counters": (I, [P, ctypes.POINTER(tadm_counters)]),
        "tadm_plan": (I, [I, I, I, I, I, ctypes.POINTER(tadm_plan_event), I, ctypes.POINTER(I)]),
        "tadm_layer_cost": (I, [I, I, I, I, I, ctypes.POINTER(I64), ctypes.POINTER(I64)]),
        "tadm_gemm": (I, [P, P, P, I, I, I, I, I, I, I, I, P]),
        "tadm_confidence": (I, [P, I, I, I, P, P, P]),
        "tadm_topk_unmask": (I, [P, I, P, P, I, I, I, I, P, P]),
        "tadm_attention": (I, [P, P, P, P, I, I, I, I, I, I, I, I, I, I, P]),
        "tadm_head_scratch_size": (I, [I, I, I, ctypes.POINTER(SZ)]),
        "tadm_head_confidence": (I, [P, P, I, I, I, I, I, P, SZ, P, P, P]),
        "tadm_head_confidence_static": (I, [P, P, I, I, I, I, I, P, P, P]),
        "tadm_probe_enable": (I, [P, I]),
        "tadm_remdm_schedule": (I, [I, I, I, ctypes.c_double, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                    ctypes.POINTER(ctypes.c_double)]),
        "tadm_remdm_uniforms": (I, [ctypes.c_uint64, I, I, I, P, P]),
        "tadm_remdm_update": (I, [P, I, P, I, I, I, I, I, I, ctypes.c_double, ctypes.c_double, ctypes.c_float,
                                  ctypes.c_uint64, I, P, P]),
        "tadm_generate_remdm": (I, [P, P, I, I, P, I, I, I, I, ctypes.c_double, ctypes.c_float, ctypes.c_uint64, P,
                                    SZ, P]),
        "tadm_eb_update": (I, [P, I, P, I, I, I, I, I, I, ctypes.c_double, ctypes.c_double, I, ctypes.c_uint64, I,
                               P, P, I, I, P, P]),
        "tadm_eb_scratch_bytes": (I, [P, I, I, I, ctypes.POINTER(SZ)]),
        "tadm_generate_entropy_bound": (I, [P, P, I, I, P, I, I, I, ctypes.c_double, ctypes.c_double,
                                            ctypes.c_double, I, ctypes.c_uint64, P, SZ, P]),
        "tadm_probe_breakdown": (I, [P, I, ctypes.POINTER(I64), ctypes.POINTER(ctypes.c_double),
                                     ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]),
        "tadm_probe_read": (I, [P, ctypes.POINTER(I64), ctypes.POINTER(ctypes.c_double),
                                ctypes.POINTER(ctypes.c_double)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(status: int, handle=None):
    if status != TADM_OK:
        msg = load_library().tadm_last_error(handle).decode() if handle else ""
        raise TadmError(status, msg)


def make_config(model) -> tadm_config:
    """tadm_config from any object with the ModelConfig attributes."""
    return tadm_config(
        vocab=model.vocab, d_model=model.d_model, n_heads=model.n_heads, n_kv_heads=model.n_kv_heads,
        head_dim=model.head_dim, ffn=model.ffn, glu=1 if model.glu == "geglu" else 0, n_shared=model.n_shared,
        n_anchor=model.n_anchor, n_denoise=model.n_denoise, fusion={"gated_mlp": 0, "paired_attn": 1, "none": 2}[model.fusion],
        fusion_rank=model.fusion_rank, fusion_heads=model.fusion_heads, dtype=1 if model.dtype == "bf16" else 0,
        tied_lm_head=int(bool(model.tied_lm_head)), norm_eps=model.norm_eps, rope_theta=model.rope_theta,
        sliding_window=getattr(model, "sliding_window", 0), global_every=getattr(model, "global_every", 0),
        qk_norm=int(bool(getattr(model, "qk_norm", False))),
        sandwich_norm=int(bool(getattr(model, "sandwich_norm", False))),
        rope_theta_global=getattr(model, "rope_theta_global", 0.0),
        qkv_split=int(bool(getattr(model, "qkv_split", False))))


# ---------------------------------------------------------------------------- C-named wrappers
def tadm_weight_inventory(cfg: tadm_config):
    lib = load_library()
    n = lib.tadm_weight_count(ctypes.byref(cfg))
    if n < 0:
        raise TadmError(1, "invalid config")
    out = []
    buf = ctypes.create_string_buffer(128)
    r, c = ctypes.c_int64(), ctypes.c_int64()
    for i in range(n):
        _check(lib.tadm_weight_info(ctypes.byref(cfg), i, buf, 128, ctypes.byref(r), ctypes.byref(c)))
        out.append((buf.value.decode(), (r.value,) if c.value == 1 else (r.value, c.value)))
    return out


def tadm_plan(prompt_len: int, gen_len: int, steps_per_block: int, K: int, block_len: int):
    lib = load_library()
    n = ctypes.c_int()
    _check(lib.tadm_plan(prompt_len, gen_len, steps_per_block, K, block_len, None, 0, ctypes.byref(n)))
    ev = (tadm_plan_event * n.value)()
    _check(lib.tadm_plan(prompt_len, gen_len, steps_per_block, K, block_len, ev, n.value, ctypes.byref(n)))
    return [(e.kind, e.block, e.n, e.k) for e in ev]


def tadm_layer_cost(L_S: int, L_A: int, L_D: int, T: int, K: int):
    full, cache = ctypes.c_int64(), ctypes.c_int64()
    _check(load_library().tadm_layer_cost(L_S, L_A, L_D, T, K, ctypes.byref(full), ctypes.byref(cache)))
    return full.value, cache.value


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream=None) -> Optional[int]:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def tadm_gemm(A, B, C, dtype: int, stream=None):
    M, K = A.shape
    N = B.shape[0]
    c_dtype = 1 if str(C.dtype) == "torch.bfloat16" else 0
    _check(load_library().tadm_gemm(_ptr(A), _ptr(B), _ptr(C), M, N, K, A.stride(0), B.stride(0), C.stride(0),
                                    dtype, c_dtype, _stream(stream)))


def tadm_confidence(logits, mask_id: int, conf, tok, stream=None):
    rows, vocab = logits.shape
    _check(load_library().tadm_confidence(_ptr(logits), rows, vocab, mask_id, _ptr(conf), _ptr(tok), _stream(stream)))


def tadm_topk_unmask(z, conf, tok, k: int, mask_id: int, selected=None, stream=None):
    batch, rows = conf.shape
    _check(load_library().tadm_topk_unmask(_ptr(z), z.stride(0), _ptr(conf), _ptr(tok), batch, rows, k, mask_id,
                                           _ptr(selected), _stream(stream)))


def tadm_head_scratch_size(rows: int, vocab: int, dtype: int) -> int:
    n = ctypes.c_size_t()
    _check(load_library().tadm_head_scratch_size(rows, vocab, dtype, ctypes.byref(n)))
    return n.value


def tadm_head_confidence(x, w, mask_id: int, conf, tok, scratch, dtype: int, stream=None):
    rows, d = x.shape
    vocab = w.shape[0]
    _check(load_library().tadm_head_confidence(_ptr(x), _ptr(w), rows, d, vocab, mask_id, dtype, _ptr(scratch),
                                               scratch.numel() * scratch.element_size(), _ptr(conf), _ptr(tok),
                                               _stream(stream)))


def tadm_head_confidence_static(x, w, mask_id: int, conf, tok, dtype: int, stream=None):
    """The same result as tadm_head_confidence, with the partials in the
    library's fixed device array instead of caller scratch (no allocation)."""
    rows, d = x.shape
    vocab = w.shape[0]
    _check(load_library().tadm_head_confidence_static(_ptr(x), _ptr(w), rows, d, vocab, mask_id, dtype, _ptr(conf),
                                                      _ptr(tok), _stream(stream)))


def tadm_attention(q, k, v, o, n_heads: int, n_kv_heads: int, rows: int, ctx: int, causal: bool, dtype: int,
                   stream=None, window: int = 0):
    batch, _, _, hd = q.shape
    kv_stride = k.shape[2]
    _check(load_library().tadm_attention(_ptr(q), _ptr(k), _ptr(v), _ptr(o), batch, n_heads, n_kv_heads, hd, rows,
                                         ctx, kv_stride, int(causal), window, dtype, _stream(stream)))


REMDM_KINDS = {"cap": 0, "loop": 1}


def tadm_remdm_schedule(kind: str, T: int, n: int, eta: float, t_on: float = 0.55, t_off: float = 0.05,
                        alpha_on: float = 0.9):
    """(alpha_t, alpha_s, sigma_t, p_unmask) of reverse step n (host only)."""
    out = (ctypes.c_double * 4)()
    _check(load_library().tadm_remdm_schedule(REMDM_KINDS[kind], T, n, eta, t_on, t_off, alpha_on, out))
    return tuple(out)


def tadm_remdm_uniforms(seed: int, step: int, batch: int, rows: int, out, stream=None):
    """The sampler's draws of a step into out (device float [batch, rows, 3])."""
    _check(load_library().tadm_remdm_uniforms(seed, step, batch, rows, _ptr(out), _stream(stream)))


def tadm_remdm_update(z, logits, first_gen: int, mask_id: int, sigma: float, p_unmask: float, top_p: float,
                      seed: int, step: int, action, stream=None):
    """One ReMDM reverse step on z [batch, rows] from logits [batch * rows, vocab]."""
    batch, rows = z.shape
    vocab = logits.shape[1]
    _check(load_library().tadm_remdm_update(_ptr(z), rows, _ptr(logits), vocab, batch, rows, first_gen, vocab,
                                            mask_id, sigma, p_unmask, top_p, seed, step, _ptr(action),
                                            _stream(stream)))



def tadm_eb_update(z, logits, first_gen: int, mask_id: int, tau: float, eta: float, last: bool, seed: int,
                   step: int, entropy, probs=None, z_sum=None, stream=None):
    """One entropy-bound step (Alg. 2) on z [batch, rows] from the logits of
    the generated positions [batch * (rows - first_gen), vocab]; entropy
    [batch * (rows - first_gen)] fp32; probs (optional, fp32 or bf16) gets
    q = exp((l - max) / tau) and z_sum (optional, fp32) Z = sum q."""
    batch, rows = z.shape
    vocab = logits.shape[1]
    p_dtype = 0
    if probs is not None:
        p_dtype = {"torch.float32": 0, "torch.bfloat16": 1}[str(probs.dtype)]
    _check(load_library().tadm_eb_update(_ptr(z), rows, _ptr(logits), vocab, batch, rows, first_gen, vocab, mask_id,
                                         tau, eta, int(bool(last)), seed, step, _ptr(entropy),
                                         _ptr(probs) if probs is not None else None, p_dtype,
                                         probs.shape[1] if probs is not None else 0, _ptr(z_sum), _stream(stream)))

# ---------------------------------------------------------------------------- model handle
class TadmModel:
    """A handle plus its torch-allocated workspace.

    ``weights`` maps inventory names to device tensors (fp32 or bf16,
    contiguous).  The handle keeps references so the memory outlives it.
    """

    def __init__(self, model, weights: Dict[str, "object"], max_batch: int, max_rows: int, max_ctx: int = 0):
        import torch
        lib = load_library()
        self.lib = lib
        self.model = model
        self.cfg = make_config(model)
        inv = tadm_weight_inventory(self.cfg)
        self.weights = []
        for name, shape in inv:
            t = weights[name]
            if tuple(t.shape) != tuple(shape) and not (len(shape) == 1 and t.numel() == shape[0]):
                raise TadmError(1, f"weight {name} has shape {tuple(t.shape)}, expected {shape}")
            if not t.is_contiguous() or not t.is_cuda:
                raise TadmError(1, f"weight {name} must be a contiguous CUDA tensor")
            self.weights.append(t)
        arr = (ctypes.c_void_p * len(self.weights))(*[t.data_ptr() for t in self.weights])
        h = ctypes.c_void_p()
        _check(lib.tadm_create(ctypes.byref(self.cfg), arr, len(self.weights), max_batch, max_rows, max_ctx,
                               ctypes.byref(h)))
        self.h = h
        n = ctypes.c_size_t()
        _check(lib.tadm_workspace_size(h, ctypes.byref(n)), h)
        self.workspace = torch.empty(max(n.value, 256), dtype=torch.uint8, device="cuda")
        _check(lib.tadm_bind_workspace(h, self.workspace.data_ptr(), n.value), h)
        self.max_batch, self.max_rows, self.max_ctx = max_batch, max_rows, max_ctx

    def close(self):
        if getattr(self, "h", None):
            self.lib.tadm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- C-named calls ----------------------------------------------------
    def tadm_cache_size(self, batch: int, rows: int) -> int:
        n = ctypes.c_size_t()
        _check(self.lib.tadm_cache_size(self.h, batch, rows, ctypes.byref(n)), self.h)
        return n.value

    def new_cache(self, batch: int, rows: int):
        import torch
        return torch.empty(self.tadm_cache_size(batch, rows), dtype=torch.uint8, device="cuda")

    def tadm_reset(self, batch: int):
        _check(self.lib.tadm_reset(self.h, batch), self.h)

    def tadm_prefill(self, prompt, stream=None):
        B, P = prompt.shape
        _check(self.lib.tadm_prefill(self.h, _ptr(prompt), B, P, _stream(stream)), self.h)

    def tadm_anchor_forward(self, x_t, t: int, h_cache, stream=None):
        B, R = x_t.shape
        _check(self.lib.tadm_anchor_forward(self.h, _ptr(x_t), B, R, t, _ptr(h_cache), _stream(stream)), self.h)

    def tadm_denoise_step(self, x_t, t: int, T: int, n_masked_at_start: int, h_cache, logits=None, conf=None,
                          tok=None, selected=None, fused=None, stream=None):
        B, R = x_t.shape
        out = tadm_step_outputs(_ptr(logits), _ptr(conf), _ptr(tok), _ptr(selected), _ptr(fused))
        _check(self.lib.tadm_denoise_step(self.h, _ptr(x_t), B, R, t, T, n_masked_at_start, _ptr(h_cache),
                                          ctypes.byref(out), _stream(stream)), self.h)

    def tadm_commit_block(self, x_block, stream=None):
        B, R = x_block.shape
        _check(self.lib.tadm_commit_block(self.h, _ptr(x_block), B, R, _stream(stream)), self.h)

    def tadm_generate(self, prompt, out, gen_len: int, steps_per_block: int, K: int, block_len: int = 0,
                      stream=None):
        B, P = prompt.shape
        _check(self.lib.tadm_generate(self.h, _ptr(prompt), B, P, _ptr(out), gen_len, steps_per_block, K,
                                      block_len, _stream(stream)), self.h)

    def tadm_generate_remdm(self, prompt, out, gen_len: int, steps: int, K: int, kind: str, eta: float,
                            top_p: float, seed: int, logits_scratch, stream=None):
        B, P = prompt.shape
        _check(self.lib.tadm_generate_remdm(self.h, _ptr(prompt), B, P, _ptr(out), gen_len, steps, K,
                                            REMDM_KINDS[kind], eta, top_p, seed, _ptr(logits_scratch),
                                            logits_scratch.numel() * logits_scratch.element_size(),
                                            _stream(stream)), self.h)

    def tadm_eb_scratch_bytes(self, batch: int, gen_len: int, self_cond: bool = True) -> int:
        out = ctypes.c_size_t(0)
        _check(self.lib.tadm_eb_scratch_bytes(self.h, batch, gen_len, int(bool(self_cond)), ctypes.byref(out)), self.h)
        return out.value

    def tadm_generate_entropy_bound(self, prompt, out, gen_len: int, steps: int, K: int, eta: float,
                                    tau_max: float, tau_min: float, seed: int, scratch, self_cond: bool = True,
                                    stream=None):
        """Alg. 2 generation; scratch: a device buffer of at least
        tadm_eb_scratch_bytes(batch, gen_len, self_cond) bytes."""
        B, P = prompt.shape
        _check(self.lib.tadm_generate_entropy_bound(self.h, _ptr(prompt), B, P, _ptr(out), gen_len, steps, K, eta,
                                                    tau_max, tau_min, int(bool(self_cond)), seed, _ptr(scratch),
                                                    scratch.numel() * scratch.element_size(), _stream(stream)),
               self.h)

    def tadm_sync_status(self):
        _check(self.lib.tadm_sync_status(self.h), self.h)

    def tadm_probe_enable(self, max_launches: int):
        _check(self.lib.tadm_probe_enable(self.h, max_launches), self.h)

    EPI_NAMES = ["plain", "residual", "qkv_rope", "glu", "fusion_gate_hidden", "fusion_out", "output_head",
                 "pa_up", "pa_silu", "pa_add", "pa_gate", "attention", "norms", "attention_short_rows"]
    N_GEMM_KINDS = 11

    def tadm_probe_breakdown(self) -> dict:
        n = len(self.EPI_NAMES)
        L, ms, fl, by = (ctypes.c_int64 * n)(), (ctypes.c_double * n)(), (ctypes.c_double * n)(), (ctypes.c_double * n)()
        _check(self.lib.tadm_probe_breakdown(self.h, n, L, ms, fl, by), self.h)
        return {self.EPI_NAMES[k]: {"launches": L[k], "ms": ms[k], "flops": fl[k], "bytes": by[k],
                                    "tflops": fl[k] / (ms[k] / 1e3) / 1e12}
                for k in range(n) if L[k] > 0}

    def tadm_probe_read(self):
        n, ms, fl = ctypes.c_int64(), ctypes.c_double(), ctypes.c_double()
        _check(self.lib.tadm_probe_read(self.h, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(fl)), self.h)
        return n.value, ms.value, fl.value

    def tadm_get_counters(self) -> dict:
        c = tadm_counters()
        _check(self.lib.tadm_get_counters(self.h, ctypes.byref(c)), self.h)
        return {f: getattr(c, f) for f, _ in tadm_counters._fields_}

    # -- user-facing ------------------------------------------------------------
    def generate(self, prompt, gen_len: int, steps_per_block: int, K: int, block_len: int = 0, stream=None):
        """Whole generation.  ``prompt`` may live on the host or the device;
        host prompts are copied in and the result copied back (pinned)."""
        import torch
        host = not prompt.is_cuda
        p = prompt.to("cuda", non_blocking=True) if host else prompt
        out = torch.empty((p.shape[0], p.shape[1] + gen_len), dtype=torch.int32, device="cuda")
        self.tadm_generate(p, out, gen_len, steps_per_block, K, block_len, stream)
        if host:
            res = torch.empty(out.shape, dtype=torch.int32, pin_memory=True)
            res.copy_(out, non_blocking=True)
            self.tadm_sync_status()
            return res
        return out


def upload_weights(model, host_weights: Dict[str, "object"]):
    """Copy generated host weights (float32 or raw bf16 bits) to the device."""
    import numpy as np
    import torch
    out = {}
    for name, w in host_weights.items():
        if w.dtype == np.uint16:
            t = torch.from_numpy(w.view(np.int16)).view(torch.bfloat16)
        else:
            t = torch.from_numpy(np.ascontiguousarray(w, dtype=np.float32))
        out[name] = t.to("cuda").contiguous()
    return out
