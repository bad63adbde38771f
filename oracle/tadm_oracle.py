"""Plain fp64 CPU oracle of TADM's anchor-cache reverse-diffusion sampling loop.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` import this module.  The CUDA library never
calls it and shares no code with it; both only consume the same seeded inputs
(``workloads``).

What it computes (paper section / equation it follows):

* Model decomposition ``c = S(z)``, ``h = A(c)``, ``x = D(Phi(c, h))``: §3.1.
* Stale-anchor fusion, general form ``h~ = h' + g * Delta``: §3.2,
  Eq. (stale-anchor-fusion).  Two instances:
    - gated residual MLP (TADM:Pretraining): App. C.2;
    - paired attention with cached shallow state (TADM:Post-train): App. C.1,
      Eqs. (paired-attention-difference) and (stale-anchor-fusion-app).
  Fusion off ("none"): the naive stale-anchor reuse baseline of App. D
  (Table naive-vs-tadm-posttrain): Alg. 1 with the fusion disabled, so the
  denoiser receives the cached anchor output itself, h~ = h'.
* Anchor-cache inference loop: Alg. 1 (Anchor-Cache Inference), §3.3;
  transformer-layer cost: Eq. (anchor-cache-compute).
* Masked-diffusion reverse step with zero-masking and carry-over unmasking:
  App. B.1.1, Eq. (mdlm-posterior-unk).
* ReMDM remasking sampler (the paper's Pretraining sampler, NEXT row):
  §5 Eq. (inf-post-TADM), App. B Eqs. (remdm-posterior, remdm-param), with
  the linear schedule, nucleus p and Cap / Loop settings of App. C.2.
* DiffusionGemma entropy-bound sampler with self-conditioning (the paper's
  Post-train sampler, NEXT row): Alg. 2 with the App. C.1 settings.
* Block diffusion with a KV cache over committed blocks (the encoder prefills
  the context causally, the decoder denoises the active block
  bidirectionally): App. C.1, "Architecture Details".
* Backbone layer: pre-norm transformer (RMSNorm, RoPE, multi-head attention
  with grouped KV heads, SwiGLU / GeGLU FFN), the layer type the workloads
  name; the paper treats it as a black box.  The Post-train backbone is
  Gemma-3 based (App. C.1 "Architecture Details", which gives no layer
  details); its Gemma-3 layer details are optional here: local layers with a
  sliding attention window and global layers with their own RoPE base in a
  fixed pattern, QK-norm, and sandwich (pre + post) norms around both
  sub-blocks.  These follow the public Gemma-3 architecture, not the paper,
  and parity for them is pinned by the special cases listed in the tests
  (window >= length reduces to full attention, window 1 to the token's own
  value, scale invariance of normalised projections).

Readings where the paper is silent:
* sampler P: confidence top-k within the active block; conf = max softmax
  probability over the vocabulary without MASK, k_n = floor((n+1)G/T) -
  floor(nG/T), ties broken toward the lower position;
* refresh at n = T - i with n mod K == 0, counter restarting per block;
* A3 LayerNorms are LayerNorm(eps 1e-6) with affine terms, GELU is the erf
  form; GeGLU uses the tanh-approximate GELU;
* A4: J = [Z, U] and F = [U; Z0; Z - Z0; M] concatenate features; the gate
  MLP hidden width is r; the mixer attention has no positional encoding;
* h_cache is the raw residual stream leaving A (no final norm);
* commit / prefill passes run S, A, Phi(c, A(c)), D fresh, with causal
  attention inside the block being committed.

All arithmetic is float64.  Weights arrive as float32 arrays or raw bf16 bit
arrays and are widened exactly.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

NEG_INF = -np.inf


# ---------------------------------------------------------------------------
# elementary ops (textbook definitions)
# ---------------------------------------------------------------------------
def widen(w: np.ndarray) -> np.ndarray:
    """Exact float64 values of a float32 or raw-bf16-bits array."""
    if w.dtype == np.uint16:
        return (w.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return w.astype(np.float64)


def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * gain, over the last axis."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def layer_norm(x: np.ndarray, w: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """(x - mean) / sqrt(var + eps) * w + b, over the last axis (biased variance)."""
    mu = np.mean(x, axis=-1, keepdims=True)
    var = np.mean((x - mu) ** 2, axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * w + b


def sigmoid(x: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-x))


def silu(x: np.ndarray) -> np.ndarray:
    return x * sigmoid(x)


try:  # library erf when available, else the scalar one from the C library
    from scipy.special import erf as _erf
except ImportError:  # pragma: no cover
    def _erf(x: np.ndarray) -> np.ndarray:
        return np.vectorize(math.erf, otypes=[np.float64])(x)


def gelu_erf(x: np.ndarray) -> np.ndarray:
    """GELU, exact form x * Phi(x) (Hendrycks & Gimpel 2016)."""
    return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))


def gelu_tanh(x: np.ndarray) -> np.ndarray:
    """GELU, tanh approximation (Hendrycks & Gimpel 2016)."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def linear(x: np.ndarray, w: np.ndarray, b: Optional[np.ndarray] = None) -> np.ndarray:
    """y = x W^T (+ b); W is [out, in]."""
    y = x @ w.T
    return y if b is None else y + b


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary position embedding, rotate-half pairing (j, j + hd/2).

    x: [H, L, hd]; pos: [L] absolute positions.
    """
    hd = x.shape[-1]
    half = hd // 2
    j = np.arange(half, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / hd)
    ang = pos.astype(np.float64)[:, None] * inv_freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, q_pos: np.ndarray, k_pos: np.ndarray,
              causal: bool, window: int = 0) -> np.ndarray:
    """softmax(q k^T / sqrt(hd)) v with grouped KV heads.

    q: [Hq, Lq, hd]; k, v: [Hkv, Lk, hd]; query head h reads KV head
    h // (Hq / Hkv).  causal: key allowed iff k_pos <= q_pos.  window > 0
    (a local layer of the Gemma-3 backbone): key allowed only if
    q_pos - k_pos < window as well.  Returns [Hq, Lq, hd].
    """
    Hq, Lq, hd = q.shape
    Hkv = k.shape[0]
    group = Hq // Hkv
    out = np.empty_like(q)
    for h in range(Hq):
        kh, vh = k[h // group], v[h // group]
        s = q[h] @ kh.T / math.sqrt(hd)
        if causal:
            s = np.where(k_pos[None, :] <= q_pos[:, None], s, NEG_INF)
        if window > 0:
            s = np.where(q_pos[:, None] - k_pos[None, :] < window, s, NEG_INF)
        s = s - np.max(s, axis=-1, keepdims=True)
        p = np.exp(s)
        p = p / np.sum(p, axis=-1, keepdims=True)
        out[h] = p @ vh
    return out


# ---------------------------------------------------------------------------
# the sampler P (confidence top-k in the active block)
# ---------------------------------------------------------------------------
def confidence(logits: np.ndarray, mask_id: int):
    """Per row: tok = argmax over v != MASK (lowest id on ties), conf = p(tok).

    Zero-masking (App. B.1.1): the MASK logit is excluded, so the model never
    predicts MASK.  conf = 1 / sum_v exp(l_v - l_max), in float64.
    """
    l = np.array(logits, dtype=np.float64, copy=True)
    l[..., mask_id] = NEG_INF
    tok = np.argmax(l, axis=-1)
    m = np.take_along_axis(l, tok[..., None], axis=-1)
    conf = 1.0 / np.sum(np.exp(l - m), axis=-1)
    return conf, tok.astype(np.int64)


def unmask_count(n: int, T: int, G: int) -> int:
    """k_n = floor((n+1) G / T) - floor(n G / T): G masked positions spread
    evenly over T steps, all of them committed by the last step."""
    return (n + 1) * G // T - n * G // T


def select_topk(z: np.ndarray, conf: np.ndarray, k: int, mask_id: int) -> np.ndarray:
    """Positions to unmask in one sequence: the k masked positions of largest
    conf, ties toward the lower position.  Carry-over (App. B.1.1): positions
    already holding a token are never candidates."""
    cand = np.nonzero(z == mask_id)[0]
    if k <= 0 or cand.size == 0:
        return np.zeros(0, dtype=np.int64)
    order = np.lexsort((cand, -conf[cand]))  # primary: conf desc, secondary: position asc
    return cand[order[:k]]


# ---------------------------------------------------------------------------
# ReMDM remasking sampler (§5 Eq. inf-post-TADM; App. B Eqs. remdm-posterior,
# remdm-param; sampler settings of App. C.2 "Sampler Details")
# ---------------------------------------------------------------------------
def remdm_alpha(t: float, kind: str, t_on: float, t_off: float, alpha_on: float) -> float:
    """alpha_t of the reverse schedule.  "cap": the linear schedule, 1 - t.
    "loop": alpha rises linearly from 0 at t = 1 to alpha_on at t_on, stays
    at alpha_on down to t_off, then rises linearly to 1 at t = 0."""
    if kind == "cap":
        return 1.0 - t
    if t > t_on:
        return alpha_on * (1.0 - t) / (1.0 - t_on)
    if t >= t_off:
        return alpha_on
    return alpha_on + (1.0 - alpha_on) * (t_off - t) / t_off


def remdm_schedule(n: int, T: int, kind: str, eta: float, t_on: float = 0.55, t_off: float = 0.05,
                   alpha_on: float = 0.9):
    """(alpha_t, alpha_s, sigma_t, p_unmask) of reverse step n = 0..T-1 from
    t = (T - n) / T to s = (T - n - 1) / T.  sigma_t is capped by
    sigma_max = min(1, (1 - alpha_s) / alpha_t), the largest value that keeps
    the posterior a distribution; "cap" uses min(eta, sigma_max) at every
    step, "loop" uses it only inside the loop phase (alpha_t = alpha_s =
    alpha_on) and 0 elsewhere.  p_unmask = (alpha_s - (1 - sigma) alpha_t) /
    (1 - alpha_t) is the probability that a masked position takes a token."""
    t = (T - n) / T
    s = (T - n - 1) / T
    a_t = remdm_alpha(t, kind, t_on, t_off, alpha_on)
    a_s = remdm_alpha(s, kind, t_on, t_off, alpha_on)
    sigma_max = min(1.0, (1.0 - a_s) / a_t) if a_t > 0.0 else 1.0
    if kind == "cap" or (t <= t_on and s >= t_off):
        sigma = min(eta, sigma_max)
    else:
        sigma = 0.0
    p_unmask = (a_s - (1.0 - sigma) * a_t) / (1.0 - a_t)
    return a_t, a_s, sigma, p_unmask


def nucleus_sample(logits: np.ndarray, mask_id: int, top_p: float, u: float) -> int:
    """One token of the nucleus (top-p) distribution of softmax(logits) over
    ids != MASK.  Nucleus N = {v : q_v >= tau}, tau the largest probability
    value such that the tokens at or above it hold >= top_p of the mass
    (tokens tied at tau are all kept).  The token is the first v of N in id
    order whose cumulative mass within N exceeds u * mass(N)."""
    l = np.asarray(logits, dtype=np.float64).copy()
    l[mask_id] = -np.inf
    q = np.exp(l - np.max(l))
    desc = np.sort(q)[::-1]
    k = int(np.searchsorted(np.cumsum(desc), top_p * q.sum(), side="left"))
    tau = desc[min(k, desc.size - 1)]
    qn = np.where(q >= tau, q, 0.0)
    c = np.cumsum(qn)
    return int(np.nonzero(c > u * c[-1])[0][0])


def remdm_step(z: np.ndarray, logits: np.ndarray, first_gen: int, sigma: float, p_unmask: float, top_p: float,
               u: np.ndarray, mask_id: int):
    """One reverse step of one sequence (Eq. inf-post-TADM).  z: [R] canvas,
    logits: [R, V], u: [R, 3] uniforms (remask, unmask, token).  Positions
    before first_gen (the prompt) never change; a generated token is remasked
    with probability sigma; a masked position unmasks with probability
    p_unmask to a nucleus sample of its logits.  Returns (z_s, action) with
    action 0 keep, 1 remask, 2 unmask."""
    out = z.copy()
    act = np.zeros(z.shape[0], dtype=np.int32)
    for r in range(first_gen, z.shape[0]):
        if z[r] != mask_id:
            if u[r, 0] < sigma:
                out[r] = mask_id
                act[r] = 1
        elif u[r, 1] < p_unmask:
            out[r] = nucleus_sample(logits[r], mask_id, top_p, u[r, 2])
            act[r] = 2
    return out, act


# ---------------------------------------------------------------------------
# DiffusionGemma entropy-bound sampler (Alg. 2, App. C.1 "Sampler Details")
# ---------------------------------------------------------------------------
def eb_temperature(n: int, T: int, tau_max: float, tau_min: float) -> float:
    """tau_n = tau_min + (tau_max - tau_min) n / T for n = T .. 1 (Alg. 2)."""
    return tau_min + (tau_max - tau_min) * n / T


def eb_row(logits: np.ndarray, tau: float, mask_id: int, u: float):
    """Per position of Alg. 2: p = softmax(l / tau) over ids != MASK, the
    argmax (ties to the lowest id), the entropy H = -sum p log p, and a draw
    from Cat(p) by inverse CDF in id order (first v whose cumulative p
    exceeds u).  Returns (p, argmax, H, draw)."""
    l = np.asarray(logits, dtype=np.float64) / tau
    l[mask_id] = -np.inf
    e = np.exp(l - np.max(l))
    p = e / e.sum()
    nz = p > 0
    H = float(-np.sum(p[nz] * np.log(p[nz])))
    c = np.cumsum(p)
    draw = int(np.nonzero(c > u * c[-1])[0][0])
    return p, int(np.argmax(p)), H, draw


def eb_accept(H: np.ndarray, eta: float) -> np.ndarray:
    """Alg. 2's accepted set: positions in ascending entropy (ties to the
    lower position), pi_m accepted when C_m - M_m <= eta, C_m the summed
    entropy of the first m and M_m their maximum (= H of pi_m)."""
    order = np.lexsort((np.arange(H.size), H))
    C = np.cumsum(H[order])
    M = np.maximum.accumulate(H[order])
    ok = np.zeros(H.size, dtype=bool)
    ok[order[C - M <= eta]] = True
    return ok


def layer_cost(L_S: int, L_A: int, L_D: int, T: int, K: int):
    """Eq. (anchor-cache-compute): (C_full, C_cache) transformer-layer calls."""
    c_full = T * (L_S + L_A + L_D)
    c_cache = T * (L_S + L_D) + (-(-T // K)) * L_A
    return c_full, c_cache


# ---------------------------------------------------------------------------
# the model
# ---------------------------------------------------------------------------
@dataclass
class _Seq:
    """Per-sequence KV context (block mode): one (K, V) pair per layer."""
    ctx_len: int = 0
    kv: Dict[str, List[np.ndarray]] = field(default_factory=dict)


class Oracle:
    """fp64 reference of the TADM networks and the Alg. 1 loop.

    ``model`` is any object with the attributes vocab, d_model, n_heads,
    n_kv_heads, head_dim, ffn, glu, n_shared, n_anchor, n_denoise, fusion,
    fusion_rank, fusion_heads, tied_lm_head, norm_eps, rope_theta.
    ``weights`` maps tensor names to arrays (float32 or raw bf16 bits).
    """

    def __init__(self, model, weights: Dict[str, np.ndarray], cache_f64_limit: int = 2 << 30):
        self.m = model
        self.mask_id = model.vocab - 1
        self._raw = weights
        total = sum(w.size for w in weights.values())
        self._keep = total * 8 <= cache_f64_limit
        self._w64: Dict[str, np.ndarray] = {}
        self.counters = {"shared": 0, "anchor": 0, "denoise": 0, "anchor_calls": 0, "steps": 0}
        self.refresh_log: List[tuple] = []

    def W(self, name: str) -> np.ndarray:
        if name in self._w64:
            return self._w64[name]
        w = widen(self._raw[name])
        if self._keep:
            self._w64[name] = w
        return w

    # -- backbone layer (pre-norm) ------------------------------------------
    def layer_index(self, name: str) -> int:
        """Position of layer "<net>.<i>." in the whole backbone: the L_S
        shared layers, then the L_A anchor layers, then the L_D denoiser
        layers."""
        net, i = name.split(".")[:2]
        first = {"shared": 0, "anchor": self.m.n_shared, "denoise": self.m.n_shared + self.m.n_anchor}[net]
        return first + int(i)

    def layer_kind(self, name: str):
        """(window, RoPE base) of a layer under the Gemma-3 pattern: layer i
        is global iff global_every > 0 and (i + 1) % global_every == 0, or
        global_every == 0.  Local layers see keys less than sliding_window
        positions back (0: all) with base rope_theta; global layers see every
        key, with base rope_theta_global (rope_theta when that is 0)."""
        m = self.m
        g = getattr(m, "global_every", 0)
        is_global = g == 0 or (self.layer_index(name) + 1) % g == 0
        if is_global:
            tg = getattr(m, "rope_theta_global", 0.0)
            return 0, (tg if tg > 0 else m.rope_theta)
        return getattr(m, "sliding_window", 0), m.rope_theta

    def layer(self, name: str, x: np.ndarray, pos: np.ndarray, seq: Optional[_Seq], causal: bool,
              keep_kv: bool) -> np.ndarray:
        """x <- x + Wo Attn(RoPE(Q), RoPE(K), V) from RMSNorm(x); then
        x <- x + Wdown (act(Wg n) * (Wu n)) with n = RMSNorm(x).

        Gemma-3 details when the model enables them: QK-norm (RMSNorm over
        head_dim of each Q and K head, gains q_norm / k_norm, before RoPE);
        sandwich norms (x <- x + RMSNorm(Wo o) with gain post_attn_norm, and
        x <- x + RMSNorm(Wdown a) with gain post_ffn_norm); the window and
        RoPE base of the layer's kind (``layer_kind``).

        Keys are the context cached in ``seq`` (committed positions) followed
        by the rows of x.  With ``keep_kv`` the rows' K, V are appended to the
        context (commit / prefill pass).
        """
        m = self.m
        hd, Hq, Hkv, F = m.head_dim, m.n_heads, m.n_kv_heads, m.ffn
        L = x.shape[0]
        window, theta = self.layer_kind(name)
        n = rms_norm(x, self.W(name + "attn_norm"), m.norm_eps)
        qkv = linear(n, self.W(name + "wqkv"))
        q = qkv[:, : Hq * hd].reshape(L, Hq, hd).transpose(1, 0, 2)
        k = qkv[:, Hq * hd: (Hq + Hkv) * hd].reshape(L, Hkv, hd).transpose(1, 0, 2)
        v = qkv[:, (Hq + Hkv) * hd:].reshape(L, Hkv, hd).transpose(1, 0, 2)
        if getattr(m, "qk_norm", False):
            q = rms_norm(q, self.W(name + "q_norm"), m.norm_eps)
            k = rms_norm(k, self.W(name + "k_norm"), m.norm_eps)
        q = rope(q, pos, theta)
        k = rope(k, pos, theta)
        if seq is not None and name in seq.kv:
            kc, vc = seq.kv[name]
            k_all = np.concatenate([kc, k], axis=1)
            v_all = np.concatenate([vc, v], axis=1)
            k_pos = np.concatenate([np.arange(kc.shape[1]), pos])
        else:
            k_all, v_all, k_pos = k, v, pos
        o = attention(q, k_all, v_all, pos, k_pos, causal, window)
        sandwich = getattr(m, "sandwich_norm", False)
        a = linear(o.transpose(1, 0, 2).reshape(L, Hq * hd), self.W(name + "wo"))
        if sandwich:
            a = rms_norm(a, self.W(name + "post_attn_norm"), m.norm_eps)
        x = x + a
        n = rms_norm(x, self.W(name + "ffn_norm"), m.norm_eps)
        gu = linear(n, self.W(name + "wgu"))
        g, u = gu[:, :F], gu[:, F:]
        act = silu(g) if m.glu == "swiglu" else gelu_tanh(g)
        f = linear(act * u, self.W(name + "wdown"))
        if sandwich:
            f = rms_norm(f, self.W(name + "post_ffn_norm"), m.norm_eps)
        x = x + f
        if keep_kv and seq is not None:
            if name in seq.kv:
                kc, vc = seq.kv[name]
                seq.kv[name] = [np.concatenate([kc, k], axis=1), np.concatenate([vc, v], axis=1)]
            else:
                seq.kv[name] = [k, v]
        return x

    def stack(self, net: str, n_layers: int, x, pos, seq, causal, keep_kv, count=True):
        for i in range(n_layers):
            x = self.layer(f"{net}.{i}.", x, pos, seq, causal, keep_kv)
        if count:
            self.counters[net] += n_layers
        return x

    # -- S, A, D (§3.1) -----------------------------------------------------
    def S(self, z: np.ndarray, pos, seq, causal=False, keep_kv=False, count=True, add=None) -> np.ndarray:
        """Shared network: token embedding (+ ``add``, the self-conditioning
        signal of Alg. 2), then L_S backbone layers."""
        c = self.W("embed")[z.astype(np.int64)]
        if add is not None:
            c = c + add
        return self.stack("shared", self.m.n_shared, c, pos, seq, causal, keep_kv, count)

    def A(self, c, pos, seq, causal=False, keep_kv=False, count=True) -> np.ndarray:
        """Anchor network: L_A backbone layers; the raw residual stream is h."""
        return self.stack("anchor", self.m.n_anchor, c, pos, seq, causal, keep_kv, count)

    def D_hidden(self, h, pos, seq, causal=False, keep_kv=False, count=True) -> np.ndarray:
        return self.stack("denoise", self.m.n_denoise, h, pos, seq, causal, keep_kv, count)

    def lm_head(self, y: np.ndarray) -> np.ndarray:
        """Final RMSNorm then the output projection (tied to the embedding when
        ``tied_lm_head``)."""
        n = rms_norm(y, self.W("final_norm"), self.m.norm_eps)
        w = self.W("embed") if self.m.tied_lm_head else self.W("lm_head")
        return linear(n, w)

    # -- fusion Phi (§3.2) ----------------------------------------------------
    def fusion_gated_mlp(self, c: np.ndarray, h: np.ndarray) -> np.ndarray:
        """App. C.2: u = [LN(c); LN(h)], g = sigmoid(W_g u + b_g),
        Delta = W_2 GELU(W_1 u + b_1) + b_2, h~ = LN(h + g * Delta)."""
        m, d, eps = self.m, self.m.d_model, self.m.norm_eps
        s = layer_norm(c, self.W("fusion.ln_c.w"), self.W("fusion.ln_c.b"), eps)
        a = layer_norm(h, self.W("fusion.ln_h.w"), self.W("fusion.ln_h.b"), eps)
        u = np.concatenate([s, a], axis=-1)
        wg1, bg1 = self.W("fusion.w_g1"), self.W("fusion.b_g1")
        g = sigmoid(linear(u, wg1[:d], bg1[:d]))
        delta = linear(gelu_erf(linear(u, wg1[d:], bg1[d:])), self.W("fusion.w2"), self.W("fusion.b2"))
        return layer_norm(h + g * delta, self.W("fusion.ln_out.w"), self.W("fusion.ln_out.b"), eps)

    def _rms_scale(self, x: np.ndarray) -> np.ndarray:
        """s_i = sqrt(mean_j x_ij^2 + eps), eps = 1e-6 (App. C.1)."""
        return np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + 1e-6)

    def mixer(self, Z: np.ndarray, U: np.ndarray) -> np.ndarray:
        """Shared mixer phi (App. C.1): J = [Z, U]; Q, K, V = J W_{Q,K,V};
        R = Z + MHA(Q, K, V) W_O; phi = R + SiLU(R W_1) W_2.  Attention is
        bidirectional over the rows of the current canvas."""
        r, H = self.m.fusion_rank, self.m.fusion_heads
        L = Z.shape[0]
        J = np.concatenate([Z, U], axis=-1)
        wqkv = self.W("fusion.wqkv")
        q = linear(J, wqkv[:r]).reshape(L, H, r // H).transpose(1, 0, 2)
        k = linear(J, wqkv[r:2 * r]).reshape(L, H, r // H).transpose(1, 0, 2)
        v = linear(J, wqkv[2 * r:]).reshape(L, H, r // H).transpose(1, 0, 2)
        pos = np.arange(L)
        o = attention(q, k, v, pos, pos, causal=False).transpose(1, 0, 2).reshape(L, r)
        R = Z + linear(o, self.W("fusion.wo"))
        return R + linear(silu(linear(R, self.W("fusion.w1"))), self.W("fusion.w2"))

    def paired_refresh(self, C0: np.ndarray, H0: np.ndarray) -> dict:
        """Quantities of App. C.1 that depend only on the refresh step:
        s_C, s_H, Z0 = (C0/s_C) W_C, U = (H0/s_H) W_H and phi(Z0, U)."""
        sC, sH = self._rms_scale(C0), self._rms_scale(H0)
        Z0 = linear(C0 / sC, self.W("fusion.wc"))
        U = linear(H0 / sH, self.W("fusion.wh"))
        return {"H0": H0, "C0": C0, "sC": sC, "sH": sH, "Z0": Z0, "U": U, "phi0": self.mixer(Z0, U)}

    def fusion_paired_attn(self, C: np.ndarray, st: dict) -> np.ndarray:
        """App. C.1: M = phi(Z, U) - phi(Z0, U)  (Eq. paired-attention-difference);
        F = [U; Z0; Z - Z0; M]; g = sigmoid(SiLU(F W_g1) W_g2 + b_g);
        H~ = H0 + g * s_H * (M W_up)  (Eq. stale-anchor-fusion-app)."""
        Z = linear(C / st["sC"], self.W("fusion.wc"))
        M = self.mixer(Z, st["U"]) - st["phi0"]
        F = np.concatenate([st["U"], st["Z0"], Z - st["Z0"], M], axis=-1)
        g = sigmoid(linear(silu(linear(F, self.W("fusion.wg1"))), self.W("fusion.wg2"), self.W("fusion.bg")))
        return st["H0"] + g * st["sH"] * linear(M, self.W("fusion.wup"))

    def make_cache(self, c: np.ndarray, h: np.ndarray):
        """What the anchor cache holds for one sequence."""
        if self.m.fusion == "paired_attn":
            return self.paired_refresh(c, h)
        return {"h": h}

    def fuse(self, c: np.ndarray, cache) -> np.ndarray:
        if self.m.fusion == "paired_attn":
            return self.fusion_paired_attn(c, cache)
        if self.m.fusion == "none":              # App. D naive reuse: D reads the stale h' as is
            return cache["h"].copy()
        return self.fusion_gated_mlp(c, cache["h"])

    # -- sessions (block mode context) ----------------------------------------
    def new_session(self, batch: int) -> List[_Seq]:
        return [_Seq() for _ in range(batch)]

    def _fresh_pass(self, seq: _Seq, z_rows: np.ndarray):
        """Causal fresh pass S -> A -> Phi(c, A(c)) -> D over rows appended to
        the context; every layer's K, V for these rows join the context."""
        L = z_rows.shape[0]
        pos = seq.ctx_len + np.arange(L)
        c = self.S(z_rows, pos, seq, causal=True, keep_kv=True, count=False)
        h = self.A(c, pos, seq, causal=True, keep_kv=True, count=False)
        ht = self.fuse(c, self.make_cache(c, h))
        self.D_hidden(ht, pos, seq, causal=True, keep_kv=True, count=False)
        seq.ctx_len += L

    def prefill(self, sess: List[_Seq], prompts: np.ndarray):
        """Encoder prefill of the prompt (block mode, App. C.1)."""
        for b, seq in enumerate(sess):
            self._fresh_pass(seq, prompts[b])

    def commit_block(self, sess: List[_Seq], z_block: np.ndarray):
        """Append a finalized block to the context (block mode, App. C.1)."""
        for b, seq in enumerate(sess):
            self._fresh_pass(seq, z_block[b])

    # -- one refresh / one denoising step of Alg. 1 -----------------------------
    def anchor_forward(self, sess: List[_Seq], z_rows: np.ndarray) -> list:
        """Refresh branch of Alg. 1: h_cache <- A(S(z)) for every sequence."""
        out = []
        for b, seq in enumerate(sess):
            pos = seq.ctx_len + np.arange(z_rows.shape[1])
            c = self.S(z_rows[b], pos, seq, count=False)
            h = self.A(c, pos, seq, count=(b == 0))
            out.append(self.make_cache(c, h))
        self.counters["anchor_calls"] += 1
        return out

    def denoise_logits(self, sess: List[_Seq], z_rows: np.ndarray, cache: list) -> np.ndarray:
        """c = S(z); h~ = Phi(c, h_cache); logits = head(D(h~)).  [B, R, V]."""
        B, R = z_rows.shape
        out = np.empty((B, R, self.m.vocab), dtype=np.float64)
        for b, seq in enumerate(sess):
            pos = seq.ctx_len + np.arange(R)
            c = self.S(z_rows[b], pos, seq, count=(b == 0))
            ht = self.fuse(c, cache[b])
            out[b] = self.lm_head(self.D_hidden(ht, pos, seq, count=(b == 0)))
        return out

    def sample(self, z_rows: np.ndarray, conf: np.ndarray, tok: np.ndarray, n: int, T: int, G: int):
        """Sampler P: unmask k_n positions per sequence.  Returns the new canvas
        and the selected positions ([B, k_n], -1 padded)."""
        k = unmask_count(n, T, G)
        z_new = z_rows.copy()
        sel = np.full((z_rows.shape[0], max(k, 0)), -1, dtype=np.int64)
        for b in range(z_rows.shape[0]):
            p = select_topk(z_rows[b], conf[b], k, self.mask_id)
            z_new[b, p] = tok[b, p]
            sel[b, : p.size] = p
        return z_new, sel

    def denoise_step(self, sess, z_rows, cache, n: int, T: int, G: int):
        """One reverse step after the (optional) refresh: logits, conf, tok and
        the sampler update.  Returns a dict."""
        logits = self.denoise_logits(sess, z_rows, cache)
        conf, tok = confidence(logits, self.mask_id)
        z_new, sel = self.sample(z_rows, conf, tok, n, T, G)
        self.counters["steps"] += 1
        return {"logits": logits, "conf": conf, "tok": tok, "z": z_new, "selected": sel}

    # -- Alg. 1 over every block -----------------------------------------------
    def generate(self, prompts: np.ndarray, gen_len: int, steps_per_block: int, K: int,
                 block_len: int = 0, step_hook=None) -> np.ndarray:
        """Alg. 1 per block.  block_len == 0: a single block over the whole
        canvas (prompt + gen_len masks, bidirectional, no KV context).
        Otherwise the prompt is prefilled, then blocks of ``block_len`` masks
        are denoised and committed one after the other."""
        B, P = prompts.shape
        mask = self.mask_id
        T = steps_per_block
        if block_len == 0:
            z = np.concatenate([prompts.astype(np.int32), np.full((B, gen_len), mask, np.int32)], axis=1)
            sess = self.new_session(B)
            z = self._run_block(sess, z, T, K, gen_len, 0, step_hook)
            return z
        assert gen_len % block_len == 0
        sess = self.new_session(B)
        self.prefill(sess, prompts.astype(np.int32))
        blocks = []
        for bi in range(gen_len // block_len):
            zb = np.full((B, block_len), mask, np.int32)
            zb = self._run_block(sess, zb, T, K, block_len, bi, step_hook)
            self.commit_block(sess, zb)
            blocks.append(zb)
        return np.concatenate([prompts.astype(np.int32)] + blocks, axis=1)

    def generate_remdm(self, prompts: np.ndarray, gen_len: int, T: int, K: int, kind: str, eta: float,
                       top_p: float, uniforms, t_on: float = 0.55, t_off: float = 0.05, alpha_on: float = 0.9,
                       step_hook=None) -> np.ndarray:
        """Alg. 1 with the ReMDM remasking sampler on one canvas (prompt +
        gen_len masks, single block): refresh when n mod K = 0, logits from
        the fused prediction, then remdm_step per sequence.  ``uniforms(n)``
        returns the [B, P + gen_len, 3] draws of step n."""
        B, P = prompts.shape
        mask = self.mask_id
        z = np.concatenate([prompts.astype(np.int32), np.full((B, gen_len), mask, np.int32)], axis=1)
        sess = self.new_session(B)
        cache = None
        for n in range(T):
            if n % K == 0:
                cache = self.anchor_forward(sess, z)
            logits = self.denoise_logits(sess, z, cache)
            _, _, sigma, p_un = remdm_schedule(n, T, kind, eta, t_on, t_off, alpha_on)
            u = uniforms(n)
            new = np.empty_like(z)
            for b in range(B):
                new[b], _ = remdm_step(z[b], logits[b], P, sigma, p_un, top_p, u[b], mask)
            if step_hook is not None:
                step_hook(n, z, logits, new)
            z = new
            self.counters["steps"] += 1
        return z

    def generate_entropy_bound(self, prompts: np.ndarray, gen_len: int, T: int, K: int, eta: float,
                               tau_max: float, tau_min: float, uniforms, self_cond: bool = True,
                               step_hook=None) -> np.ndarray:
        """Alg. 2 (DiffusionGemma entropy-bound sampling) with the anchor
        cache of Alg. 1 on one canvas (prompt + gen_len generated positions,
        single block).  The canvas starts as uniform noise over ids != MASK;
        step i = 0 .. T-1 is Alg. 2's n = T - i: refresh when i mod K = 0,
        logits of the fused prediction with the self-conditioning signal s
        added to the input embedding of the generated positions, p, argmax,
        entropy and a draw per position, s <- p E; for n > 1 accepted
        positions take their draw and the others fresh noise; n = 1 returns
        the argmax canvas.  ``uniforms(i)`` gives [B, P + gen_len, 3] draws of
        step i (draw, noise token, unused); step T gives the initial noise.
        ``step_hook(n, z, new_z, H)`` sees each step's canvas before and after
        and the entropies of the generated positions."""
        B, P = prompts.shape
        V, mask, d = self.m.vocab, self.mask_id, self.m.d_model
        L = P + gen_len
        pos = np.arange(L)
        E = self.W("embed")
        u = uniforms(T)
        z = np.concatenate([prompts.astype(np.int32),
                            np.floor(u[:, P:, 1] * (V - 1)).astype(np.int32)], axis=1)
        s = np.zeros((B, L, d))
        cache = [None] * B
        for i in range(T):
            n = T - i
            if i % K == 0:
                for b in range(B):
                    c = self.S(z[b], pos, None, count=False, add=s[b])
                    cache[b] = self.make_cache(c, self.A(c, pos, None, count=(b == 0)))
                self.counters["anchor_calls"] += 1
            tau = eb_temperature(n, T, tau_max, tau_min)
            u = uniforms(i)
            new_z, new_s, Hs = z.copy(), np.zeros_like(s), np.zeros((B, gen_len))
            for b in range(B):
                c = self.S(z[b], pos, None, count=(b == 0), add=s[b])
                logits = self.lm_head(self.D_hidden(self.fuse(c, cache[b]), pos, None, count=(b == 0)))
                H, draw, am = np.zeros(gen_len), np.zeros(gen_len, np.int32), np.zeros(gen_len, np.int32)
                for g in range(gen_len):
                    p, am[g], H[g], draw[g] = eb_row(logits[P + g], tau, mask, u[b, P + g, 0])
                    new_s[b, P + g] = p @ E
                if n > 1:
                    noise = np.floor(u[b, P:, 1] * (V - 1)).astype(np.int32)
                    new_z[b, P:] = np.where(eb_accept(H, eta), draw, noise)
                else:
                    new_z[b, P:] = am
                Hs[b] = H
            if step_hook is not None:
                step_hook(n, z, new_z, Hs)
            z = new_z
            s = new_s if self_cond else np.zeros_like(s)
            self.counters["steps"] += 1
        return z

    def _run_block(self, sess, z, T, K, G, block_idx, step_hook):
        cache = None
        for n in range(T):           # n = T - i, i = T .. 1
            if n % K == 0:           # Alg. 1 refresh test (T - i) mod K = 0
                cache = self.anchor_forward(sess, z)
                self.refresh_log.append((block_idx, n))
            r = self.denoise_step(sess, z, cache, n, T, G)
            if step_hook is not None:
                step_hook(block_idx, n, z, r)
            z = r["z"]
        return z
