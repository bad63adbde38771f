"""Seeded synthetic workloads for the TADM anchor-cache sampling loop.

This module is the one piece that both sides of the parity check share: the
workload presets (model dimensions, batch, prompt and generation lengths,
schedule) and the seeded generators of random-init weights and prompt token
ids.  It holds no step of the method's arithmetic; it only draws numbers.

Weights: every tensor is N(mean, std^2) from Philox4x32-10 + Box-Muller
(Salmon et al., SC'11), keyed by (seed, tensor index, element index), rounded
to bf16 (round-to-nearest-even) for bf16 workloads.  Matrices use std 0.02;
norm gains are 1 and biases 0 unless ``affine_std`` asks for random ones (the
tests use that to exercise the affine terms).  The paper zero-initialises the
fusion output projections for training; here every fusion matrix is random
so that the fusion arithmetic is exercised.

Prompts: uniform ids over [0, V-2] or Zipf(1.1) ranks r in [1, V-1] mapped to
id r-1 by inverse-CDF sampling; the id V-1 is reserved for MASK.

Matrix layout convention: a projection from n_in to n_out features is stored
as [n_out, n_in] (row j holds the weights of output feature j), and
``y = x @ W.T``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None
_LIB_LOCK = threading.Lock()

PROMPT_STREAM = 0x50524F4D  # stream id of prompt draws ("PROM")
REMDM_STREAM = 0x52454D44   # stream id of the ReMDM sampler's draws ("REMD")


# --------------------------------------------------------------------------
# native generator (plain C, OpenMP)
# --------------------------------------------------------------------------
def build_generator(force: bool = False) -> str:
    """Compile workloads/philox.c into an in-tree shared object."""
    src = os.path.join(_HERE, "philox.c")
    so = os.path.join(_HERE, "_philox.so")
    if force or not os.path.exists(so) or os.path.getmtime(so) < os.path.getmtime(src):
        tmp = so + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-o", tmp, src, "-lm"])
        os.replace(tmp, so)
    return so


def _lib():
    global _LIB
    with _LIB_LOCK:
        if _LIB is None:
            lib = ctypes.CDLL(build_generator())
            u64, u32, i64 = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int64
            lib.wl_philox4x32_10.argtypes = [ctypes.POINTER(u32), ctypes.POINTER(u32), ctypes.POINTER(u32)]
            lib.wl_philox_u32.argtypes = [u64, u32, i64, ctypes.c_void_p]
            lib.wl_philox_blocks.argtypes = [u64, u32, u64, i64, ctypes.c_void_p]
            lib.wl_normal_f32.argtypes = [u64, u32, i64, ctypes.c_double, ctypes.c_double, ctypes.c_void_p]
            lib.wl_normal_bf16.argtypes = [u64, u32, i64, ctypes.c_double, ctypes.c_double, ctypes.c_void_p]
            _LIB = lib
    return _LIB


def philox4x32_10(ctr, key) -> Tuple[int, int, int, int]:
    """One Philox4x32-10 block (the published known-answer vectors pin this)."""
    c = (ctypes.c_uint32 * 4)(*ctr)
    k = (ctypes.c_uint32 * 2)(*key)
    o = (ctypes.c_uint32 * 4)()
    _lib().wl_philox4x32_10(c, k, o)
    return tuple(int(v) for v in o)


def philox_u32(seed: int, stream: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint32)
    if n:
        _lib().wl_philox_u32(seed, stream, n, out.ctypes.data)
    return out


def philox_blocks(seed: int, stream: int, first_block: int, n_blocks: int) -> np.ndarray:
    """uint32 [n_blocks, 4]: the words of Philox blocks first_block .. (counter =
    (block lo, block hi, stream, 0), key = (seed lo, seed hi))."""
    out = np.empty((n_blocks, 4), dtype=np.uint32)
    if n_blocks:
        _lib().wl_philox_blocks(seed, stream, first_block, n_blocks, out.ctypes.data)
    return out


def remdm_uniforms(seed: int, step: int, batch: int, rows: int) -> np.ndarray:
    """float64 [batch, rows, 3]: the ReMDM sampler's three uniforms in [0, 1)
    for every canvas position of reverse step ``step`` (remask, unmask, token).
    Position (b, r) of step n uses Philox block (n * batch + b) * rows + r of
    REMDM_STREAM; uniform j = (word j >> 8) * 2^-24."""
    w = philox_blocks(seed, REMDM_STREAM, (step * batch) * rows, batch * rows)
    return ((w[:, :3] >> 8).astype(np.float64) * (1.0 / 16777216.0)).reshape(batch, rows, 3)


def normal(seed: int, stream: int, n: int, mean: float, std: float, dtype: str) -> np.ndarray:
    """``n`` draws of N(mean, std^2); dtype 'f32' -> float32, 'bf16' -> uint16 bf16 bits."""
    if dtype == "f32":
        out = np.empty(n, dtype=np.float32)
        if n:
            _lib().wl_normal_f32(seed, stream, n, mean, std, out.ctypes.data)
    elif dtype == "bf16":
        out = np.empty(n, dtype=np.uint16)
        if n:
            _lib().wl_normal_bf16(seed, stream, n, mean, std, out.ctypes.data)
    else:
        raise ValueError(dtype)
    return out


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of raw bf16 bits to float32."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# model / workload presets
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class ModelConfig:
    vocab: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    glu: str = "swiglu"          # "swiglu" (SiLU gate) | "geglu" (tanh-GELU gate)
    n_shared: int = 0            # L_S: transformer layers inside S (embedding always)
    n_anchor: int = 4            # L_A
    n_denoise: int = 2           # L_D
    fusion: str = "gated_mlp"    # "gated_mlp" (Pretraining) | "paired_attn" (Post-train) | "none" (stale reuse, no fusion)
    fusion_rank: int = 256       # r of the paired-attention fusion
    fusion_heads: int = 4
    dtype: str = "bf16"          # "f32" | "bf16"
    tied_lm_head: bool = False
    norm_eps: float = 1e-6
    rope_theta: float = 10000.0
    # Gemma-3 backbone details (off by default): local layers attend to keys
    # less than `sliding_window` positions back (0: unbounded); layer i of the
    # whole backbone (S, then A, then D) is global iff global_every > 0 and
    # (i + 1) % global_every == 0, and every layer is global when
    # global_every == 0; global layers use rope_theta_global (0: rope_theta);
    # qk_norm: RMSNorm over head_dim of every Q and K head before RoPE;
    # sandwich_norm: RMSNorm of each sub-block's output before the residual add
    sliding_window: int = 0
    global_every: int = 0
    rope_theta_global: float = 0.0
    qk_norm: bool = False
    sandwich_norm: bool = False
    # precision of the GPU path (the oracle is exact either way): the QKV
    # projections take their input as bf16 hi + lo
    qkv_split: bool = False

    @property
    def mask_id(self) -> int:
        return self.vocab - 1


@dataclass(frozen=True)
class Workload:
    name: str
    model: ModelConfig
    batch: int
    prompt_len: int
    gen_len: int
    steps_per_block: int
    K: int
    block_len: int = 0           # 0: one block over the whole canvas (no KV cache)
    prompt_dist: str = "zipf"    # "uniform" | "zipf"
    seed: int = 0
    k_sweep: Tuple[int, ...] = ()

    @property
    def n_blocks(self) -> int:
        return 1 if self.block_len == 0 else self.gen_len // self.block_len

    @property
    def total_len(self) -> int:
        return self.prompt_len + self.gen_len


TINY = ModelConfig(vocab=1024, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=1024,
                   n_anchor=4, n_denoise=2, dtype="f32")
# the bf16 presets carry the QKV projections' input as bf16 hi + lo (qkv_split): the
# attention logits are the backbone's most rounding-sensitive quantity
SMALL = ModelConfig(vocab=32768, d_model=768, n_heads=12, n_kv_heads=12, head_dim=64, ffn=3072,
                    n_anchor=8, n_denoise=4, qkv_split=True)
BLOCK = ModelConfig(vocab=128000, d_model=2048, n_heads=16, n_kv_heads=8, head_dim=128, ffn=8192,
                    n_anchor=16, n_denoise=6, qkv_split=True)
POSTTRAIN = ModelConfig(vocab=262144, d_model=5376, n_heads=32, n_kv_heads=16, head_dim=128, ffn=21504,
                        glu="geglu", n_shared=2, n_anchor=54, n_denoise=6, fusion="paired_attn",
                        tied_lm_head=True, qkv_split=True)
# the same backbone with the Gemma-3 layer details: 5 local layers (1024-key
# sliding window, RoPE base 1e4) per global layer (RoPE base 1e6), QK-norm and
# sandwich norms
POSTTRAIN_G3 = replace(POSTTRAIN, sliding_window=1024, global_every=6, rope_theta_global=1e6, qk_norm=True,
                       sandwich_norm=True)

WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload("tiny", TINY, batch=1, prompt_len=32, gen_len=96, steps_per_block=32, K=4,
                     prompt_dist="uniform", k_sweep=(1, 4)),
    "small": Workload("small", SMALL, batch=16, prompt_len=256, gen_len=768, steps_per_block=128, K=4,
                      k_sweep=(1, 4)),
    "block": Workload("block", BLOCK, batch=32, prompt_len=512, gen_len=1536, steps_per_block=16, K=4,
                      block_len=32, k_sweep=(1, 2, 4, 8)),
    "posttrain": Workload("posttrain", POSTTRAIN, batch=8, prompt_len=1024, gen_len=1024,
                          steps_per_block=32, K=4, block_len=32, k_sweep=(1, 4)),
    "sweep": Workload("sweep", BLOCK, batch=32, prompt_len=512, gen_len=2048, steps_per_block=16, K=4,
                      block_len=32, k_sweep=(1, 2, 4, 8, 16)),
    "posttrain_g3": Workload("posttrain_g3", POSTTRAIN_G3, batch=8, prompt_len=1024, gen_len=1024,
                             steps_per_block=32, K=4, block_len=32, k_sweep=(1, 4)),
    # the post-training sampler settings of App. C.1: one 256-token canvas after the prompt, 48 reverse
    # steps, anchor refresh K in {1, 2, 3}
    "posttrain_canvas": Workload("posttrain_canvas", POSTTRAIN, batch=8, prompt_len=256, gen_len=256,
                                 steps_per_block=48, K=2, k_sweep=(1, 2, 3)),
}


def get_workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    model_over = {k[6:]: v for k, v in overrides.items() if k.startswith("model_")}
    top_over = {k: v for k, v in overrides.items() if not k.startswith("model_")}
    if model_over:
        w = replace(w, model=replace(w.model, **model_over))
    if top_over:
        w = replace(w, **top_over)
    return w


# --------------------------------------------------------------------------
# weight inventory: names, shapes and init statistics
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class TensorSpec:
    name: str
    shape: Tuple[int, ...]
    kind: str  # "matrix" | "gain" | "bias"


def weight_specs(m: ModelConfig) -> List[TensorSpec]:
    """Ordered list of every parameter tensor of the model."""
    d, hd, F = m.d_model, m.head_dim, m.ffn
    nqkv = (m.n_heads + 2 * m.n_kv_heads) * hd
    specs = [TensorSpec("embed", (m.vocab, d), "matrix")]
    for net, n in (("shared", m.n_shared), ("anchor", m.n_anchor), ("denoise", m.n_denoise)):
        for i in range(n):
            p = f"{net}.{i}."
            specs += [
                TensorSpec(p + "attn_norm", (d,), "gain"),
                TensorSpec(p + "wqkv", (nqkv, d), "matrix"),      # rows: Q heads, K heads, V heads
            ]
            if m.qk_norm:
                specs += [TensorSpec(p + "q_norm", (hd,), "gain"), TensorSpec(p + "k_norm", (hd,), "gain")]
            specs.append(TensorSpec(p + "wo", (d, m.n_heads * hd), "matrix"))
            if m.sandwich_norm:
                specs.append(TensorSpec(p + "post_attn_norm", (d,), "gain"))
            specs += [
                TensorSpec(p + "ffn_norm", (d,), "gain"),
                TensorSpec(p + "wgu", (2 * F, d), "matrix"),      # rows: gate (F), then up (F)
                TensorSpec(p + "wdown", (d, F), "matrix"),
            ]
            if m.sandwich_norm:
                specs.append(TensorSpec(p + "post_ffn_norm", (d,), "gain"))
    if m.fusion == "gated_mlp":
        specs += [
            TensorSpec("fusion.ln_c.w", (d,), "gain"), TensorSpec("fusion.ln_c.b", (d,), "bias"),
            TensorSpec("fusion.ln_h.w", (d,), "gain"), TensorSpec("fusion.ln_h.b", (d,), "bias"),
            # rows [0, d): W_g ; rows [d, 5d): W_1  (both read u = [LN(c); LN(h)], 2d wide)
            TensorSpec("fusion.w_g1", (5 * d, 2 * d), "matrix"),
            TensorSpec("fusion.b_g1", (5 * d,), "bias"),      # [b_g ; b_1]
            TensorSpec("fusion.w2", (d, 4 * d), "matrix"),
            TensorSpec("fusion.b2", (d,), "bias"),
            TensorSpec("fusion.ln_out.w", (d,), "gain"), TensorSpec("fusion.ln_out.b", (d,), "bias"),
        ]
    elif m.fusion == "paired_attn":
        r = m.fusion_rank
        specs += [
            TensorSpec("fusion.wc", (r, d), "matrix"),
            TensorSpec("fusion.wh", (r, d), "matrix"),
            TensorSpec("fusion.wqkv", (3 * r, 2 * r), "matrix"),   # rows: W_Q, W_K, W_V
            TensorSpec("fusion.wo", (r, r), "matrix"),
            TensorSpec("fusion.w1", (2 * r, r), "matrix"),
            TensorSpec("fusion.w2", (r, 2 * r), "matrix"),
            TensorSpec("fusion.wg1", (r, 4 * r), "matrix"),
            TensorSpec("fusion.wg2", (1, r), "matrix"),
            TensorSpec("fusion.bg", (1,), "bias"),
            TensorSpec("fusion.wup", (d, r), "matrix"),
        ]
    elif m.fusion != "none":
        raise ValueError(m.fusion)
    specs.append(TensorSpec("final_norm", (d,), "gain"))
    if not m.tied_lm_head:
        specs.append(TensorSpec("lm_head", (m.vocab, d), "matrix"))
    return specs


def make_weights(m: ModelConfig, seed: int = 0, std: float = 0.02, affine_std: float = 0.0,
                 only: Optional[List[str]] = None) -> Dict[str, np.ndarray]:
    """Generate every weight tensor.

    Returns float32 arrays for f32 models and uint16 bf16 bit arrays for bf16
    models (use :func:`as_f32` for an exact float32 view of the values).
    """
    out = {}
    for tid, s in enumerate(weight_specs(m)):
        if only is not None and s.name not in only:
            continue
        n = int(np.prod(s.shape))
        if s.kind == "matrix":
            mean, sd = 0.0, std
        elif s.kind == "gain":
            mean, sd = 1.0, affine_std
        else:
            mean, sd = 0.0, affine_std
        out[s.name] = normal(seed, tid, n, mean, sd, m.dtype).reshape(s.shape)
    return out


def as_f32(w: np.ndarray) -> np.ndarray:
    """Exact float32 values of a generated tensor (bf16 bits are widened)."""
    if w.dtype == np.uint16:
        return bf16_bits_to_f32(w)
    return w.astype(np.float32, copy=False)


# --------------------------------------------------------------------------
# prompts
# --------------------------------------------------------------------------
def _zipf_cdf(n_ranks: int, s: float) -> np.ndarray:
    w = np.arange(1, n_ranks + 1, dtype=np.float64) ** (-s)
    c = np.cumsum(w)
    return c / c[-1]


def make_prompts(w: Workload, batch: Optional[int] = None, seed: Optional[int] = None) -> np.ndarray:
    """int32 [batch, prompt_len] prompt ids in [0, V-2] (V-1 is MASK)."""
    B = w.batch if batch is None else batch
    seed = w.seed if seed is None else seed
    V, P = w.model.vocab, w.prompt_len
    raw = philox_u32(seed, PROMPT_STREAM, B * P)
    u = (raw >> 8).astype(np.float64) * (1.0 / 16777216.0)
    if w.prompt_dist == "uniform":
        ids = np.floor(u * (V - 1)).astype(np.int64)
    elif w.prompt_dist == "zipf":
        cdf = _zipf_cdf(V - 1, 1.1)
        ids = np.searchsorted(cdf, u, side="right").astype(np.int64)  # rank-1
    else:
        raise ValueError(w.prompt_dist)
    ids = np.minimum(ids, V - 2)
    return ids.reshape(B, P).astype(np.int32)


def initial_canvas(w: Workload, prompts: np.ndarray) -> np.ndarray:
    """int32 [B, P+G]: prompt followed by MASK everywhere else."""
    B = prompts.shape[0]
    z = np.full((B, w.total_len), w.model.mask_id, dtype=np.int32)
    z[:, : w.prompt_len] = prompts
    return z


def random_canvas(w: Workload, batch: int, rows: int, mask_frac: float, seed: int,
                  start: int = 0) -> np.ndarray:
    """A partially unmasked canvas for teacher-forced single-step checks.

    Positions ``< start`` are never masked (they model the prompt).  Each other
    position is MASK with probability ``mask_frac``, else a uniform id.
    """
    V = w.model.vocab
    raw = philox_u32(seed, 0x43414E56, 2 * batch * rows).reshape(2, batch, rows)
    ids = ((raw[0] >> 8).astype(np.float64) * (1.0 / 16777216.0) * (V - 1)).astype(np.int64)
    um = (raw[1] >> 8).astype(np.float64) * (1.0 / 16777216.0)
    z = np.minimum(ids, V - 2).astype(np.int32)
    masked = um < mask_frac
    masked[:, :start] = False
    z[masked] = w.model.mask_id
    return z
