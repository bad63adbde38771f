"""Pins of the CPU oracle against things the paper and mathematics fix.

No GPU.  Each test pins one part of ``oracle/`` against a closed form, a
library routine, a value printed in the paper (``tests/golden``), an
invariant of the method, or brute force on a tiny input.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

import workloads as wl
from oracle import tadm_oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


def tiny_model(**kw):
    base = dict(vocab=64, d_model=32, n_heads=4, n_kv_heads=2, head_dim=8, ffn=48, n_shared=0,
                n_anchor=2, n_denoise=1, dtype="f32", fusion="gated_mlp", fusion_rank=16, fusion_heads=4)
    base.update(kw)
    return wl.ModelConfig(**base)


def tiny_oracle(seed=3, affine_std=0.1, std=0.2, **kw):
    m = tiny_model(**kw)
    return O.Oracle(m, wl.make_weights(m, seed=seed, std=std, affine_std=affine_std))


# --------------------------------------------------------------------------- generator
def test_philox_known_answers():
    kat = json.load(open(os.path.join(GOLD, "philox_kat.json")))
    for v in kat["vectors"]:
        ctr = [int(x, 16) for x in v["ctr"]]
        key = [int(x, 16) for x in v["key"]]
        assert wl.philox4x32_10(ctr, key) == tuple(int(x, 16) for x in v["out"])


def test_generator_moments_and_bf16_rounding():
    x = wl.normal(7, 11, 1 << 20, 0.0, 0.02, "f32").astype(np.float64)
    assert abs(x.mean()) < 1e-4 and abs(x.std() - 0.02) < 1e-4
    b = wl.normal(7, 11, 4096, 0.0, 0.02, "bf16")
    f = wl.normal(7, 11, 4096, 0.0, 0.02, "f32")
    # bf16 is the round-to-nearest-even of the float32 draw
    wide = wl.bf16_bits_to_f32(b).astype(np.float64)
    assert np.all(np.abs(wide - f) <= np.abs(wide) * 2.0 ** -8)   # within half a bf16 ulp
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ref, b)                                  # torch's conversion is also RNE


def test_zipf_prompts_follow_the_power_law():
    """Prompt ids (the synthetic stand-in for real prompts): rank r = id + 1
    with p(r) proportional to r^-1.1 over ranks 1 .. V-1; the empirical
    frequencies of the first ranks match it and MASK never appears."""
    m = tiny_model(vocab=1000)
    w = wl.Workload("z", m, batch=64, prompt_len=4096, gen_len=8, steps_per_block=1, K=1, prompt_dist="zipf")
    ids = wl.make_prompts(w, seed=9).ravel()
    assert ids.min() >= 0 and ids.max() <= m.vocab - 2
    r = np.arange(1, m.vocab, dtype=np.float64)
    p = r ** -1.1 / np.sum(r ** -1.1)
    f = np.bincount(ids, minlength=m.vocab - 1)[: m.vocab - 1] / ids.size
    se = np.sqrt(p[:20] * (1 - p[:20]) / ids.size)
    assert np.all(np.abs(f[:20] - p[:20]) < 5 * se), (f[:5], p[:5])


# --------------------------------------------------------------------------- elementary ops
def test_norms_against_torch_and_closed_form():
    x = rng.standard_normal((5, 12))
    g, b = rng.standard_normal(12), rng.standard_normal(12)
    ref = Fn.layer_norm(torch.from_numpy(x), (12,), torch.from_numpy(g), torch.from_numpy(b), 1e-6)
    np.testing.assert_allclose(O.layer_norm(x, g, b, 1e-6), ref.numpy(), rtol=1e-12, atol=1e-12)
    ref = Fn.rms_norm(torch.from_numpy(x), (12,), torch.from_numpy(g), 1e-6)
    np.testing.assert_allclose(O.rms_norm(x, g, 1e-6), ref.numpy(), rtol=1e-12, atol=1e-12)
    # constant row c: RMSNorm -> sign(c) * gain * |c|/sqrt(c^2 + eps)
    c = -3.0
    out = O.rms_norm(np.full((1, 4), c), np.array([1.0, 2.0, 3.0, 4.0]), 1e-6)
    np.testing.assert_allclose(out[0], -np.array([1, 2, 3, 4]) * 3.0 / math.sqrt(9 + 1e-6), rtol=1e-14)
    # hand example: LayerNorm of [1, 2, 3, 4]: mean 2.5, var 1.25
    ln = O.layer_norm(np.array([[1.0, 2.0, 3.0, 4.0]]), np.ones(4), np.zeros(4), 0.0)
    np.testing.assert_allclose(ln[0], np.array([-1.5, -0.5, 0.5, 1.5]) / math.sqrt(1.25), rtol=1e-14)


def test_activations_against_torch():
    x = np.linspace(-6, 6, 101)
    t = torch.from_numpy(x)
    np.testing.assert_allclose(O.gelu_erf(x), Fn.gelu(t).numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.gelu_tanh(x), Fn.gelu(t, approximate="tanh").numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.silu(x), Fn.silu(t).numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.sigmoid(x), torch.sigmoid(t).numpy(), rtol=1e-12, atol=1e-14)


def test_rope_complex_form_and_relative_property():
    hd, L = 16, 7
    x = rng.standard_normal((3, L, hd))
    pos = np.array([0, 1, 5, 9, 100, 1000, 4095])
    out = O.rope(x, pos, 10000.0)
    # complex form: (x_j + i x_{j+hd/2}) * exp(i * pos * theta^(-2j/hd))
    z = x[..., : hd // 2] + 1j * x[..., hd // 2:]
    freq = 10000.0 ** (-np.arange(hd // 2) * 2.0 / hd)
    zr = z * np.exp(1j * pos[:, None] * freq[None, :])
    np.testing.assert_allclose(out, np.concatenate([zr.real, zr.imag], -1), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.rope(x, np.zeros(L, int), 1e4), x)   # position 0 is the identity
    # dot products depend only on the position difference
    q, k = rng.standard_normal((1, 1, hd)), rng.standard_normal((1, 1, hd))
    d1 = (O.rope(q, np.array([7]), 1e4) * O.rope(k, np.array([3]), 1e4)).sum()
    d2 = (O.rope(q, np.array([104]), 1e4) * O.rope(k, np.array([100]), 1e4)).sum()
    assert abs(d1 - d2) < 1e-12


@pytest.mark.parametrize("causal", [False, True])
def test_attention_against_sdpa(causal):
    Hq, Hkv, L, hd = 4, 2, 9, 8
    q = rng.standard_normal((Hq, L, hd))
    k = rng.standard_normal((Hkv, L, hd))
    v = rng.standard_normal((Hkv, L, hd))
    pos = np.arange(L)
    out = O.attention(q, k, v, pos, pos, causal)
    kk = torch.from_numpy(k).repeat_interleave(Hq // Hkv, 0)
    vv = torch.from_numpy(v).repeat_interleave(Hq // Hkv, 0)
    ref = Fn.scaled_dot_product_attention(torch.from_numpy(q), kk, vv, is_causal=causal)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_brute_force_scalar_loops():
    Hq, Hkv, Lq, Lk, hd = 2, 1, 3, 5, 4
    q = rng.standard_normal((Hq, Lq, hd))
    k = rng.standard_normal((Hkv, Lk, hd))
    v = rng.standard_normal((Hkv, Lk, hd))
    qp, kp = np.array([2, 3, 4]), np.arange(Lk)
    out = O.attention(q, k, v, qp, kp, causal=True)
    for h in range(Hq):
        for i in range(Lq):
            w = [math.exp(sum(q[h, i, t] * k[0, j, t] for t in range(hd)) / 2.0) if j <= qp[i] else 0.0
                 for j in range(Lk)]
            s = sum(w)
            for t in range(hd):
                assert abs(out[h, i, t] - sum(w[j] * v[0, j, t] for j in range(Lk)) / s) < 1e-12


# --------------------------------------------------------------------------- backbone layer
def _layer_parts(o, name):
    m = o.m
    hd, Hq, Hkv = m.head_dim, m.n_heads, m.n_kv_heads
    W = o.W
    return (W(name + "wqkv")[: Hq * hd], W(name + "wqkv")[Hq * hd:(Hq + Hkv) * hd],
            W(name + "wqkv")[(Hq + Hkv) * hd:])


def test_layer_single_token_closed_form():
    """One token at position 0: RoPE is the identity and attention returns V,
    so the layer is x + Wo expand(Wv n1) + Wdown(act(Wg n2) * Wu n2)."""
    for glu in ("swiglu", "geglu"):
        o = tiny_oracle(glu=glu)
        m = o.m
        x = rng.standard_normal((1, m.d_model))
        out = o.layer("anchor.0.", x, np.array([0]), None, causal=False, keep_kv=False)
        _, _, wv = _layer_parts(o, "anchor.0.")
        n1 = O.rms_norm(x, o.W("anchor.0.attn_norm"), m.norm_eps)
        v = (n1 @ wv.T).reshape(m.n_kv_heads, m.head_dim)
        attn = np.repeat(v, m.n_heads // m.n_kv_heads, axis=0).reshape(1, -1)   # head h reads KV h // group
        x1 = x + attn @ o.W("anchor.0.wo").T
        n2 = O.rms_norm(x1, o.W("anchor.0.ffn_norm"), m.norm_eps)
        wgu = o.W("anchor.0.wgu")
        gate, up = n2 @ wgu[: m.ffn].T, n2 @ wgu[m.ffn:].T
        act = O.silu(gate) if glu == "swiglu" else O.gelu_tanh(gate)
        np.testing.assert_allclose(out, x1 + (act * up) @ o.W("anchor.0.wdown").T, rtol=1e-12, atol=1e-12)


def test_layer_shift_invariance_and_causal_prefix():
    o = tiny_oracle()
    x = rng.standard_normal((6, o.m.d_model))
    a = o.layer("anchor.1.", x, np.arange(6), None, False, False)
    b = o.layer("anchor.1.", x, np.arange(6) + 37, None, False, False)
    np.testing.assert_allclose(a, b, rtol=1e-10, atol=1e-10)        # RoPE is relative
    c1 = o.layer("anchor.1.", x, np.arange(6), None, True, False)
    c2 = o.layer("anchor.1.", x[:4], np.arange(4), None, True, False)
    np.testing.assert_allclose(c1[:4], c2, rtol=1e-12, atol=1e-12)  # causal rows ignore later rows
    assert not np.allclose(a[:4], c1[:4])


def test_gqa_equals_mha_with_repeated_kv_heads():
    og = tiny_oracle(n_heads=4, n_kv_heads=2)
    mm = tiny_model(n_heads=4, n_kv_heads=4)
    w = dict(og._raw)
    hd, d = 8, 32
    wqkv = og.W("anchor.0.wqkv")
    q, k, v = wqkv[:32], wqkv[32:48], wqkv[48:64]
    rep = lambda t: np.repeat(t.reshape(2, hd, d), 2, axis=0).reshape(4 * hd, d)
    w["anchor.0.wqkv"] = np.concatenate([q, rep(k), rep(v)]).astype(np.float32)
    om = O.Oracle(mm, w)
    x = rng.standard_normal((5, d))
    np.testing.assert_allclose(og.layer("anchor.0.", x, np.arange(5), None, False, False),
                               om.layer("anchor.0.", x, np.arange(5), None, False, False), rtol=1e-12, atol=1e-12)


def test_kv_context_equals_one_causal_pass():
    """Prefill + commit through the KV cache equals one causal fresh pass over
    the concatenated rows (block-mode encoder, App. C.1)."""
    o = tiny_oracle(n_shared=1)
    z = rng.integers(0, 63, size=11).astype(np.int32)
    s1 = o.new_session(1)[0]
    o._fresh_pass(s1, z[:7])
    o._fresh_pass(s1, z[7:])
    s2 = o.new_session(1)[0]
    o._fresh_pass(s2, z)
    for name in s1.kv:
        np.testing.assert_allclose(s1.kv[name][0], s2.kv[name][0], rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(s1.kv[name][1], s2.kv[name][1], rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------- fusion (App. C.2)
def test_gated_mlp_zero_weights_closed_form():
    """W = 0, b_g = beta_g, b_2 = beta: g = sigmoid(beta_g), Delta = beta,
    h~ = LN(h + sigmoid(beta_g) * beta)."""
    o = tiny_oracle(affine_std=0.0)
    d = o.m.d_model
    w = dict(o._raw)
    w["fusion.w_g1"] = np.zeros_like(w["fusion.w_g1"])
    w["fusion.w2"] = np.zeros_like(w["fusion.w2"])
    bg = rng.standard_normal(5 * d).astype(np.float32)
    b2 = rng.standard_normal(d).astype(np.float32)
    w["fusion.b_g1"], w["fusion.b2"] = bg, b2
    o2 = O.Oracle(o.m, w)
    c, h = rng.standard_normal((3, d)), rng.standard_normal((3, d))
    exp = O.layer_norm(h + O.sigmoid(bg[:d].astype(np.float64)) * b2, np.ones(d), np.zeros(d), 1e-6)
    np.testing.assert_allclose(o2.fusion_gated_mlp(c, h), exp, rtol=1e-12, atol=1e-12)


def test_gated_mlp_gate_and_hidden_rows():
    """With W2 = I-like selection the output isolates g * GELU(W1 u + b1):
    checks which rows are the gate and which the hidden projection."""
    o = tiny_oracle(affine_std=0.0)
    d = o.m.d_model
    w = dict(o._raw)
    w2 = np.zeros((d, 4 * d), np.float32)
    w2[np.arange(d), np.arange(d)] = 1.0            # Delta_j = GELU(hidden_j)
    w["fusion.w2"] = w2
    w["fusion.b2"] = np.zeros(d, np.float32)
    o2 = O.Oracle(o.m, w)
    c, h = rng.standard_normal((2, d)), rng.standard_normal((2, d))
    u = np.concatenate([O.layer_norm(c, 1, 0, 1e-6), O.layer_norm(h, 1, 0, 1e-6)], -1)
    wg1, bg1 = o2.W("fusion.w_g1"), o2.W("fusion.b_g1")
    g = O.sigmoid(u @ wg1[:d].T + bg1[:d])
    hid = O.gelu_erf(u @ wg1[d:2 * d].T + bg1[d:2 * d])
    np.testing.assert_allclose(o2.fusion_gated_mlp(c, h), O.layer_norm(h + g * hid, 1, 0, 1e-6), rtol=1e-11, atol=1e-12)


# --------------------------------------------------------------------------- fusion (App. C.1)
def paired_oracle(**kw):
    return tiny_oracle(fusion="paired_attn", n_shared=1, tied_lm_head=True, **kw)


def test_paired_attention_identity_at_fresh_anchor():
    """C = C0 implies M = 0 and H~ = H0 exactly (App. C.1)."""
    o = paired_oracle()
    C0, H0 = rng.standard_normal((6, 32)), rng.standard_normal((6, 32))
    st = o.paired_refresh(C0, H0)
    out = o.fusion_paired_attn(C0.copy(), st)
    assert np.array_equal(out, H0)
    C = C0 + 0.3 * rng.standard_normal((6, 32))
    assert not np.allclose(o.fusion_paired_attn(C, st), H0)


def test_paired_attention_zero_up_projection():
    o = paired_oracle()
    w = dict(o._raw)
    w["fusion.wup"] = np.zeros_like(w["fusion.wup"])
    o2 = O.Oracle(o.m, w)
    C0, H0 = rng.standard_normal((5, 32)), rng.standard_normal((5, 32))
    st = o2.paired_refresh(C0, H0)
    np.testing.assert_array_equal(o2.fusion_paired_attn(rng.standard_normal((5, 32)), st), H0)


def test_paired_attention_uniform_mixer_closed_form():
    """W_Q = W_K = 0 makes every attention row uniform, so MHA returns the
    column mean of V = J W_V; with W_1 = 0 the FFN vanishes, hence
    phi(Z, U) = Z + mean_rows(J W_V) W_O, and with W_g1 = 0 the gate is
    sigmoid(b_g).  Then H~ = H0 + sigmoid(b_g) s_H (M W_up) in closed form."""
    o = paired_oracle()
    r = o.m.fusion_rank
    w = dict(o._raw)
    wqkv = w["fusion.wqkv"].copy()
    wqkv[: 2 * r] = 0.0
    w["fusion.wqkv"] = wqkv
    w["fusion.w1"] = np.zeros_like(w["fusion.w1"])
    w["fusion.wg1"] = np.zeros_like(w["fusion.wg1"])
    w["fusion.bg"] = np.array([0.7], np.float32)
    o2 = O.Oracle(o.m, w)
    W = o2.W
    L = 5
    C0, H0, C = (rng.standard_normal((L, 32)) for _ in range(3))
    sC = np.sqrt((C0 ** 2).mean(-1, keepdims=True) + 1e-6)
    sH = np.sqrt((H0 ** 2).mean(-1, keepdims=True) + 1e-6)
    Z0, Z, U = (C0 / sC) @ W("fusion.wc").T, (C / sC) @ W("fusion.wc").T, (H0 / sH) @ W("fusion.wh").T
    wv = W("fusion.wqkv")[2 * r:]

    def phi(Zx):
        V = np.concatenate([Zx, U], -1) @ wv.T
        return Zx + np.repeat(V.mean(0, keepdims=True), L, 0) @ W("fusion.wo").T

    M = phi(Z) - phi(Z0)
    exp = H0 + O.sigmoid(float(np.float32(0.7))) * sH * (M @ W("fusion.wup").T)
    st = o2.paired_refresh(C0, H0)
    np.testing.assert_allclose(o2.fusion_paired_attn(C, st), exp, rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------- sampler P
def test_confidence_hand_values():
    V = 6
    l = np.log(np.array([[1.0, 2.0, 2.0, 1.0, 1.0, 50.0]]))   # MASK (id 5) would win: excluded
    conf, tok = O.confidence(l, mask_id=V - 1)
    assert tok[0] == 1                                          # tie between ids 1, 2 -> lower id
    assert abs(conf[0] - 2.0 / 7.0) < 1e-15
    conf, tok = O.confidence(np.zeros((2, V)), V - 1)
    np.testing.assert_allclose(conf, 1.0 / (V - 1))
    assert np.all(tok == 0)


def test_topk_brute_force_and_carry_over():
    mask = 9
    for trial in range(200):
        L = int(rng.integers(1, 20))
        z = np.where(rng.random(L) < 0.6, mask, rng.integers(0, 9, L))
        conf = rng.choice([0.1, 0.2, 0.3, 0.5], size=L)             # many ties
        k = int(rng.integers(0, L + 2))
        got = O.select_topk(z, conf, k, mask)
        cand = [p for p in range(L) if z[p] == mask]
        want = sorted(cand, key=lambda p: (-conf[p], p))[:k]
        assert list(got) == want
        assert all(z[p] == mask for p in got)


def test_unmask_schedule():
    for G, T, k in ((96, 32, 3), (768, 128, 6), (32, 16, 2), (32, 32, 1), (7, 3, None), (5, 8, None)):
        ks = [O.unmask_count(n, T, G) for n in range(T)]
        assert sum(ks) == G and min(ks) >= 0
        if k is not None:
            assert ks == [k] * T


def test_layer_cost_against_tables_1_and_2():
    g = json.load(open(os.path.join(GOLD, "layer_cost.json")))
    for row in g["table1_ratio"]:
        full, cache = O.layer_cost(row["L_S"], row["L_A"], row["L_D"], row["T"], row["K"])
        assert round(cache / full, 2) == row["ratio_2dp"]
    for row in g["table2_calls"]:
        _, tadm = O.layer_cost(0, 12, 6, row["T"], row["K"])
        mdlm, _ = O.layer_cost(0, 0, 12, row["T"], 1)
        assert tadm == row["tadm"] and mdlm == row["mdlm"]
        assert round(tadm / mdlm, 2) == row["ratio_2dp"]


# --------------------------------------------------------------------------- Alg. 1 loop
def _gen(o, K, block_len=0, P=5, G=12, T=4, hook=None):
    prompts = rng.integers(0, o.m.vocab - 1, size=(2, P)).astype(np.int32)
    return prompts, o.generate(prompts, G, T, K, block_len, step_hook=hook)


def test_refresh_schedule_and_count():
    for K in (1, 2, 3, 4, 5):
        o = tiny_oracle()
        T, nblk = 6, 2
        _gen(o, K, block_len=4, G=8, T=T)
        assert o.refresh_log == [(b, n) for b in range(nblk) for n in range(T) if n % K == 0]
        assert o.counters["anchor_calls"] == nblk * (-(-T // K))
        assert o.counters["anchor"] == nblk * (-(-T // K)) * o.m.n_anchor
        assert o.counters["denoise"] == nblk * T * o.m.n_denoise


def test_k1_is_single_stage_dlm():
    """K = 1 refreshes at every step, so each step is one fresh pass
    D(Phi(c, A(c))): rebuild that loop directly and compare trajectories."""
    o = tiny_oracle()
    prompts, z1 = _gen(o, K=1, G=9, T=3)
    z = np.concatenate([prompts, np.full((2, 9), o.mask_id, np.int32)], 1)
    for n in range(3):
        logits = np.stack([o.lm_head(o.D_hidden(o.fusion_gated_mlp(c, o.A(c, np.arange(14), None)),
                                                np.arange(14), None))
                           for c in (o.S(z[b], np.arange(14), None) for b in range(2))])
        conf, tok = O.confidence(logits, o.mask_id)
        for b in range(2):
            p = O.select_topk(z[b], conf[b], O.unmask_count(n, 3, 9), o.mask_id)
            z[b, p] = tok[b, p]
    np.testing.assert_array_equal(z, z1)


@pytest.mark.parametrize("fusion,block_len", [("gated_mlp", 0), ("gated_mlp", 4), ("paired_attn", 4)])
def test_carry_over_zero_masking_and_stale_cache(fusion, block_len):
    o = tiny_oracle(fusion=fusion, n_shared=1 if fusion == "paired_attn" else 0,
                    tied_lm_head=fusion == "paired_attn")
    seen = []

    def hook(b, n, z, r):
        assert np.all(r["tok"] != o.mask_id)                       # zero-masking
        fixed = z != o.mask_id
        assert np.array_equal(r["z"][fixed], z[fixed])             # carry-over
        assert np.sum((z == o.mask_id) & (r["z"] != o.mask_id)) == 2 * O.unmask_count(n, 4, 4 if block_len else 12)
        seen.append((b, n))

    prompts, z = _gen(o, K=3, block_len=block_len, hook=hook)
    assert np.all(z != o.mask_id)
    np.testing.assert_array_equal(z[:, :5], prompts)
    assert len(seen) == (3 if block_len else 1) * 4


def test_stale_anchor_is_reused_between_refreshes():
    """Between refreshes the fusion reads the cached h of the refresh step
    (Alg. 1): the step-1 logits of K=2 equal D(Phi(S(z_1), A(S(z_0))))."""
    o = tiny_oracle()
    logs = {}
    prompts, _ = _gen(o, K=2, G=8, T=4, hook=lambda b, n, z, r: logs.setdefault(n, (z.copy(), r["logits"])))
    z0, _ = logs[0]
    z1, l1 = logs[1]
    L = z0.shape[1]
    pos = np.arange(L)
    for b in range(2):
        h0 = o.A(o.S(z0[b], pos, None), pos, None)
        want = o.lm_head(o.D_hidden(o.fusion_gated_mlp(o.S(z1[b], pos, None), h0), pos, None))
        np.testing.assert_allclose(l1[b], want, rtol=1e-12, atol=1e-12)


def test_paired_attention_gate_features():
    """A gate MLP that reads one feature of the Z - Z0 block of F:
    W_g1 row 0 selects column 2r (first feature of Z - Z0), W_g2 = [alpha, 0..],
    so g = sigmoid(alpha * SiLU((Z - Z0)_0) + b_g) per row, recovered from
    (H~ - H0) / (s_H * (M W_up))."""
    o = paired_oracle()
    r = o.m.fusion_rank
    w = dict(o._raw)
    wg1 = np.zeros((r, 4 * r), np.float32)
    wg1[0, 2 * r] = 1.0
    wg2 = np.zeros((1, r), np.float32)
    wg2[0, 0] = 1.5
    w["fusion.wg1"], w["fusion.wg2"], w["fusion.bg"] = wg1, wg2, np.array([-0.25], np.float32)
    o2 = O.Oracle(o.m, w)
    L = 6
    C0, H0 = rng.standard_normal((L, 32)), rng.standard_normal((L, 32))
    C = C0 + rng.standard_normal((L, 32))
    st = o2.paired_refresh(C0, H0)
    out = o2.fusion_paired_attn(C, st)
    sC = np.sqrt((C0 ** 2).mean(-1, keepdims=True) + 1e-6)
    dz0 = ((C - C0) / sC) @ o2.W("fusion.wc")[0]
    g = 1.0 / (1.0 + np.exp(-(1.5 * dz0 / (1.0 + np.exp(-dz0)) - 0.25)))
    Z = (C / sC) @ o2.W("fusion.wc").T
    MW = (o2.mixer(Z, st["U"]) - st["phi0"]) @ o2.W("fusion.wup").T
    np.testing.assert_allclose((out - H0) / (st["sH"] * MW), np.repeat(g[:, None], 32, 1), rtol=1e-8)


def test_tied_head_reads_the_embedding():
    """Tied output head: logits = RMSNorm(y) E^T, so for y = E[t] the
    self inner product wins and the argmax is t."""
    m = tiny_model(fusion="paired_attn", n_shared=1, tied_lm_head=True, d_model=64, vocab=128)
    o = O.Oracle(m, wl.make_weights(m, seed=5, std=0.2))
    assert "lm_head" not in o._raw
    E = o.W("embed")
    logits = o.lm_head(E[:127])
    assert np.array_equal(np.argmax(logits, -1), np.arange(127))


# --------------------------------------------------------------------- fusion off (App. D)
def test_fusion_off_is_one_backbone_at_a_refresh():
    """Fusion off (the naive stale-reuse baseline of App. D): at a refresh step
    D reads A's output unchanged, so anchor (a layers) + denoiser (b layers)
    is one stack of a + b layers.  Rebuild it as a model with no anchor layers
    whose denoiser holds the same a + b layers, and compare logits exactly."""
    o = tiny_oracle(fusion="none", n_anchor=2, n_denoise=2)
    m2 = tiny_model(fusion="none", n_anchor=0, n_denoise=4)
    w2 = {}
    for k, v in o._raw.items():
        if k.startswith("anchor."):
            w2["denoise." + k[len("anchor."):]] = v
        elif k.startswith("denoise."):
            i, rest = k[len("denoise."):].split(".", 1)
            w2[f"denoise.{int(i) + 2}.{rest}"] = v
        else:
            w2[k] = v
    assert set(w2) == {s.name for s in wl.weight_specs(m2)}
    o2 = O.Oracle(m2, w2)
    z = rng.integers(0, o.m.vocab - 1, (2, 7)).astype(np.int32)
    z[:, 3:] = o.mask_id
    l1 = o.denoise_logits(o.new_session(2), z, o.anchor_forward(o.new_session(2), z))
    l2 = o2.denoise_logits(o2.new_session(2), z, o2.anchor_forward(o2.new_session(2), z))
    np.testing.assert_array_equal(l1, l2)


def test_fusion_off_ignores_the_current_canvas():
    """With fusion off the denoiser sees only the cached h': logits between
    refreshes do not depend on the current canvas; with the gated-MLP fusion
    they do (the current state enters through c)."""
    for fusion, same in (("none", True), ("gated_mlp", False)):
        o = tiny_oracle(fusion=fusion)
        z0 = rng.integers(0, o.m.vocab - 1, (2, 6)).astype(np.int32)
        z0[:, 2:] = o.mask_id
        z1 = z0.copy()
        z1[:, 2:4] = rng.integers(0, o.m.vocab - 1, (2, 2))
        cache = o.anchor_forward(o.new_session(2), z0)
        l0 = o.denoise_logits(o.new_session(2), z0, cache)
        l1 = o.denoise_logits(o.new_session(2), z1, cache)
        assert np.array_equal(l0, l1) == same


# --------------------------------------------------------------------- ReMDM sampler (NEXT row)
def test_remdm_sigma_zero_is_masked_diffusion_posterior():
    """sigma_t = 0 recovers the masked-diffusion posterior (App. B, after Eq.
    remdm-posterior): with the linear schedule a masked position unmasks with
    probability (alpha_s - alpha_t) / (1 - alpha_t) = 1 / (T - n), and no
    token is ever remasked."""
    T = 17
    for n in range(T):
        a_t, a_s, sigma, p_un = O.remdm_schedule(n, T, "cap", 0.0)
        assert sigma == 0.0
        assert abs(p_un - 1.0 / (T - n)) < 1e-14
        assert abs(a_t - n / T) < 1e-15 and abs(a_s - (n + 1) / T) < 1e-15
    z = np.array([5, 9, 63, 63, 2, 63], np.int32)
    u = np.full((6, 3), 0.0)
    out, act = O.remdm_step(z, rng.standard_normal((6, 64)), 1, 0.0, 0.0, 0.9, u, 63)
    assert np.array_equal(out, z) and not act.any()


@pytest.mark.parametrize("kind,eta,T", [("cap", 0.04, 128), ("cap", 0.5, 9), ("loop", 0.02, 1024), ("loop", 0.02, 64)])
def test_remdm_posterior_is_a_distribution(kind, eta, T):
    """For every step both cases of Eq. remdm-posterior are distributions
    (sigma within [0, sigma_max]) and the last step unmasks everything."""
    for n in range(T):
        a_t, a_s, sigma, p_un = O.remdm_schedule(n, T, kind, eta)
        stay = (1.0 - a_s - sigma * a_t) / (1.0 - a_t)
        assert 0.0 <= sigma <= 1.0 and 0.0 <= a_t <= a_s <= 1.0
        assert -1e-12 <= p_un <= 1.0 + 1e-12 and stay >= -1e-12
        assert abs(p_un + stay - 1.0) < 1e-12
    _, a_s, sigma, p_un = O.remdm_schedule(T - 1, T, kind, eta)
    assert a_s == 1.0 and sigma == 0.0 and abs(p_un - 1.0) < 1e-12


def test_remdm_loop_phase_holds_alpha_on():
    """ReMDM-Loop: alpha is alpha_on throughout the loop phase, where sigma =
    eta; there the expected masked fraction 1 - alpha_on is a fixed point of
    one step (unmasking and remasking balance); no remasking outside it."""
    T, eta, a_on = 400, 0.02, 0.9
    inside = 0
    for n in range(T):
        t, s = (T - n) / T, (T - n - 1) / T
        a_t, a_s, sigma, p_un = O.remdm_schedule(n, T, "loop", eta, 0.55, 0.05, a_on)
        if t <= 0.55 and s >= 0.05:
            inside += 1
            assert a_t == a_s == a_on and sigma == eta
            m = 1.0 - a_on
            assert abs(m * (1.0 - p_un) + (1.0 - m) * sigma - m) < 1e-12
        else:
            assert sigma == 0.0
    assert inside == round((0.55 - 0.05) * T)


def test_nucleus_sample_brute_force():
    """Inverse-CDF sampling within the nucleus: on a grid of u the token
    frequencies are the renormalised nucleus probabilities, the nucleus is
    the smallest set of most probable tokens reaching top_p (built here by a
    sorted walk), and MASK is never drawn."""
    logits = np.array([0.3, 2.0, -1.0, 1.2, 2.0, 0.9, 5.0, 1.5])   # id 7 is MASK (largest after 6)
    mask, top_p = 6, 0.8
    q = np.exp(logits - logits[np.arange(8) != mask].max())
    q[mask] = 0.0
    order = sorted(range(8), key=lambda v: -q[v])
    keep, acc = [], 0.0
    for v in order:
        if acc >= top_p * q.sum() and q[v] < q[keep[-1]]:
            break
        keep.append(v)
        acc += q[v]
    want = np.zeros(8)
    want[keep] = q[keep] / q[keep].sum()
    grid = (np.arange(20000) + 0.5) / 20000
    got = np.bincount([O.nucleus_sample(logits, mask, top_p, u) for u in grid], minlength=8) / grid.size
    assert got[mask] == 0.0
    np.testing.assert_allclose(got, want, atol=1e-4)


def test_nucleus_top_p_one_is_plain_categorical():
    lg = rng.standard_normal(50)
    q = np.exp(lg - lg.max())
    q[49] = 0.0
    c = np.cumsum(q) / q.sum()
    for u in rng.random(200):
        assert O.nucleus_sample(lg, 49, 1.0, u) == int(np.searchsorted(c, u, side="right"))


def test_remdm_step_rates_and_prompt():
    """Monte Carlo over the shared Philox draws: generated tokens are
    remasked at rate sigma, masked positions unmask at rate p_unmask, the
    prompt never changes and unmasked tokens come from the nucleus."""
    V, R, P, mask = 32, 4000, 100, 31
    z = np.where(rng.random(R) < 0.5, mask, rng.integers(0, 31, R)).astype(np.int32)
    lg = rng.standard_normal((R, V))
    u = wl.remdm_uniforms(11, 3, 1, R)[0]
    out, act = O.remdm_step(z, lg, P, 0.3, 0.6, 0.9, u, mask)
    assert np.array_equal(out[:P], z[:P])
    gen = np.arange(R) >= P
    tok, msk = gen & (z != mask), gen & (z == mask)
    r1, r2 = (act[tok] == 1).mean(), (act[msk] == 2).mean()
    assert abs(r1 - 0.3) < 4 * np.sqrt(0.3 * 0.7 / tok.sum()) and abs(r2 - 0.6) < 4 * np.sqrt(0.24 / msk.sum())
    assert np.all(out[act == 2] != mask) and np.all(out[act == 1] == mask)


def test_remdm_uniforms_follow_philox():
    """The sampler's draws: block (n * B + b) * R + r of the REMD stream,
    uniform j = (word j >> 8) * 2^-24."""
    u = wl.remdm_uniforms(77, 5, 3, 11)
    for b, r in ((0, 0), (2, 10), (1, 4)):
        blk = (5 * 3 + b) * 11 + r
        w = wl.philox4x32_10([blk & 0xFFFFFFFF, blk >> 32, wl.REMDM_STREAM, 0], [77, 0])
        assert list(u[b, r]) == [(w[j] >> 8) / 16777216.0 for j in range(3)]


def test_remdm_uniform_roles_and_edges():
    """u[:, 0] alone decides remasking, u[:, 1] alone unmasking, u[:, 2] the
    token; u = 0 draws the first nucleus token in id order (never a token of
    zero nucleus mass)."""
    mask = 9
    z = np.array([1, 2, mask, mask], np.int32)
    lg = np.zeros((4, 10))
    lg[:, 7] = 6.0                      # token 7 alone holds 0.98 > 0.9 of the mass
    u = np.array([[0.0, 0.99, 0.5], [0.99, 0.0, 0.5], [0.0, 0.99, 0.5], [0.99, 0.0, 0.0]])
    out, act = O.remdm_step(z, lg, 0, 0.5, 0.5, 0.9, u, mask)
    assert list(act) == [1, 0, 0, 2] and list(out) == [mask, 2, mask, 7]
    assert O.nucleus_sample(lg[0], mask, 0.9, 0.0) == 7


def test_remdm_loop_alpha_is_continuous():
    """The Loop time warp is continuous: alpha(1) = 0, alpha(t_on) = alpha_on
    from both sides, alpha(t_off) = alpha_on, alpha(0) = 1."""
    f = lambda t: O.remdm_alpha(t, "loop", 0.55, 0.05, 0.9)  # noqa: E731
    assert f(1.0) == 0.0 and f(0.0) == 1.0
    for t in (0.55, 0.05):
        assert abs(f(t + 1e-9) - 0.9) < 1e-7 and abs(f(t - 1e-9) - 0.9) < 1e-7


def test_remdm_token_uses_its_own_uniform():
    """The token of an unmasking position is drawn with u[:, 2]: two equally
    likely tokens 3 and 7, u[:, 1] = 0.1 (unmask) and u[:, 2] = 0.9 give 7."""
    lg = np.full((1, 10), -30.0)
    lg[0, 3] = lg[0, 7] = 0.0
    out, act = O.remdm_step(np.array([9], np.int32), lg, 0, 0.0, 0.5, 0.9, np.array([[0.99, 0.1, 0.9]]), 9)
    assert act[0] == 2 and out[0] == 7


# ---------------------------------------------------------- entropy-bound sampler (Alg. 2, NEXT row)
def test_eb_temperature_is_linear_between_the_limits():
    T = 48
    assert O.eb_temperature(T, T, 0.8, 0.4) == 0.8 and abs(O.eb_temperature(0, T, 0.8, 0.4) - 0.4) < 1e-15
    d = [O.eb_temperature(n, T, 0.8, 0.4) - O.eb_temperature(n - 1, T, 0.8, 0.4) for n in range(1, T + 1)]
    assert np.allclose(d, 0.4 / T, atol=1e-15)


def test_eb_row_closed_forms():
    """Uniform logits: p uniform over the V-1 ids != MASK and H = log(V-1);
    argmax ties go to the lowest id; a dominant logit gives H -> 0; the draws
    on a grid of u reproduce p (inverse CDF in id order)."""
    V, mask = 9, 8
    p, am, H, _ = O.eb_row(np.zeros(V), 0.7, mask, 0.3)
    assert np.allclose(p[:mask], 1 / 8) and p[mask] == 0.0 and am == 0 and abs(H - np.log(8)) < 1e-12
    lg = np.zeros(V)
    lg[5] = 60.0
    assert O.eb_row(lg, 0.5, mask, 0.9)[2] < 1e-30 and O.eb_row(lg, 0.5, mask, 0.9)[1] == 5
    lg = rng.standard_normal(V)
    p = O.eb_row(lg, 0.6, mask, 0.0)[0]
    q = np.exp(lg[:mask] / 0.6 - (lg[:mask] / 0.6).max())
    assert np.allclose(p[:mask], q / q.sum())
    grid = (np.arange(20000) + 0.5) / 20000
    got = np.bincount([O.eb_row(lg, 0.6, mask, u)[3] for u in grid], minlength=V) / grid.size
    assert np.allclose(got, p, atol=1e-4)


def test_eb_accept_against_a_direct_loop():
    """Accepted set of Alg. 2 by brute force: walk the positions in ascending
    entropy and accept a position while the entropy of the ones before it
    sums to at most eta; at least the lowest-entropy position is accepted."""
    assert list(O.eb_accept(np.array([0.2, 0.2, 0.2]), 0.1)) == [True, False, False]
    assert list(O.eb_accept(np.array([0.05, 0.01, 0.3, 0.02]), 0.1)) == [True, True, True, True]
    for _ in range(50):
        H = rng.random(30) * rng.choice([0.01, 0.1, 1.0])
        eta = rng.choice([0.0, 0.05, 0.5])
        want = np.zeros(30, bool)
        acc = 0.0
        for r in sorted(range(30), key=lambda i: (H[i], i)):
            if acc <= eta:
                want[r] = True
            acc += H[r]
        assert np.array_equal(O.eb_accept(H, eta), want)


def test_eb_one_step_is_the_argmax_of_the_noise_canvas():
    """T = 1 (n = 1 only): the output is the argmax of the fused prediction
    on the initial noise canvas, which the test rebuilds from the network."""
    o = tiny_oracle()
    P, G, V = 3, 5, o.m.vocab
    prompts = rng.integers(0, V - 1, (2, P)).astype(np.int32)
    draws = lambda i: wl.remdm_uniforms(3, i, 2, P + G)  # noqa: E731
    out = o.generate_entropy_bound(prompts, G, 1, 1, 0.1, 0.8, 0.4, draws)
    u = draws(1)
    for b in range(2):
        z = np.concatenate([prompts[b], np.floor(u[b, P:, 1] * (V - 1)).astype(np.int32)])
        pos = np.arange(P + G)
        c = o.S(z, pos, None)
        logits = o.lm_head(o.D_hidden(o.fuse(c, o.make_cache(c, o.A(c, pos, None))), pos, None))
        assert np.array_equal(out[b, P:], np.argmax(np.where(np.arange(V) == o.mask_id, -np.inf, logits[P:]), -1))
        assert np.array_equal(out[b, :P], prompts[b])


def test_eb_unbounded_accepts_every_draw_and_refreshes_per_alg1():
    """eta = inf accepts every position, so before the last step the canvas
    is the categorical draws; the anchor refreshes ceil(T / K) times."""
    o = tiny_oracle()
    P, G = 2, 4
    prompts = np.array([[1, 2]], np.int32)
    seen = []
    draws = lambda i: (seen.append(i), wl.remdm_uniforms(9, i, 1, P + G))[1]  # noqa: E731
    o.counters["anchor_calls"] = 0
    out = o.generate_entropy_bound(prompts, G, 5, 2, np.inf, 0.8, 0.4, draws)
    assert o.counters["anchor_calls"] == 3 and seen == [5, 0, 1, 2, 3, 4]
    assert out.shape == (1, P + G) and np.all(out != o.mask_id)


def test_eb_draw_intervals_are_half_open():
    """Cat(p) by inverse CDF: id v owns [c_{v-1}, c_v), so u on an edge
    belongs to the next id (uniform p = 1/8, exact binary fractions)."""
    lg = np.zeros(9)
    assert [O.eb_row(lg, 1.0, 8, u)[3] for u in (0.0, 0.124, 0.125, 0.25, 0.875, 0.9999)] == [0, 0, 1, 2, 7, 7]


def test_eb_rejected_positions_are_renoised_uniformly():
    """eta < 0 accepts nothing: every generated position of a step n > 1
    becomes floor(u1 (V - 1)) of that step's draws, an id != MASK, and the
    prompt stays; with eta = inf every position keeps its categorical draw."""
    o = tiny_oracle()
    P, G, V = 2, 6, o.m.vocab
    prompts = np.array([[3, 4]], np.int32)
    draws = lambda i: wl.remdm_uniforms(21, i, 1, P + G)  # noqa: E731
    seen = []
    o.generate_entropy_bound(prompts, G, 3, 1, -1.0, 0.8, 0.4, draws,
                             step_hook=lambda n, z, new, H: seen.append((n, new.copy(), H.copy())))
    assert [n for n, _, _ in seen] == [3, 2, 1]
    for i, (n, new, H) in enumerate(seen[:2]):
        want = np.floor(draws(i)[0, P:, 1] * (V - 1)).astype(np.int32)
        assert np.array_equal(new[0, P:], want) and np.array_equal(new[0, :P], prompts[0])
        assert np.all(H >= 0) and np.all(H <= np.log(V - 1) + 1e-12)


def test_eb_self_conditioning_feeds_p_E_into_the_next_step():
    """T = 2, K = 2, eta = inf: step n = 2 runs on the noise canvas with s = 0
    and every position takes its draw; step n = 1 (tau = 0.6) embeds that
    canvas plus s = p_2 E, reuses the anchor cache of step n = 2 and returns
    the argmax.  Without self-conditioning the second step sees s = 0.  The
    entropies of step n = 1 carry the difference (the argmax may not)."""
    o = tiny_oracle()
    P, G, V = 2, 5, o.m.vocab
    prompts = np.array([[7, 1]], np.int32)
    draws = lambda i: wl.remdm_uniforms(33, i, 1, P + G)  # noqa: E731
    pos, E = np.arange(P + G), o.W("embed")
    z = np.concatenate([prompts[0], np.floor(draws(2)[0, P:, 1] * (V - 1)).astype(np.int32)])
    c = o.S(z, pos, None)
    cache = o.make_cache(c, o.A(c, pos, None))
    lg = o.lm_head(o.D_hidden(o.fuse(c, cache), pos, None))
    s = np.zeros((P + G, o.m.d_model))
    for g in range(G):
        p, _, _, z[P + g] = O.eb_row(lg[P + g], 0.8, o.mask_id, draws(0)[0, P + g, 0])
        s[P + g] = p @ E
    H1 = {}
    for sc, add in ((True, s), (False, None)):
        c = o.S(z, pos, None, add=add)
        lg = o.lm_head(o.D_hidden(o.fuse(c, cache), pos, None))
        rows = [O.eb_row(lg[P + g], 0.6, o.mask_id, 0.5) for g in range(G)]
        H1[sc] = np.array([r[2] for r in rows])
        seen = []
        got = o.generate_entropy_bound(prompts, G, 2, 2, np.inf, 0.8, 0.4, draws, self_cond=sc,
                                       step_hook=lambda n, z0, new, H: seen.append((n, H.copy())))
        assert np.array_equal(got[0, P:], [r[1] for r in rows]), sc
        assert [n for n, _ in seen] == [2, 1] and np.allclose(seen[1][1][0], H1[sc], rtol=1e-12, atol=0), sc
    assert np.max(np.abs(H1[True] - H1[False])) > 1e-6


def test_eb_signal_enters_as_an_embedding_offset():
    """The self-conditioning signal is added to the token embedding: adding
    E[v] - E[z_l] at position l gives the shared network's output for the
    canvas with z_l replaced by v."""
    o = tiny_oracle()
    z = np.array([1, 5, 9, 2, 4], np.int32)
    pos, E = np.arange(5), o.W("embed")
    add = np.zeros((5, o.m.d_model))
    add[3] = E[11] - E[2]
    z2 = z.copy()
    z2[3] = 11
    assert np.allclose(o.S(z, pos, None, add=add), o.S(z2, pos, None), rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------ output head, block-mode context
def test_output_head_normalises_the_hidden_state():
    """logits = RMSNorm(y) W_out^T: a constant row y = a 1 normalises to
    sign(a) gain, so its logits are sign(a) (W_out gain)_v in closed form,
    and scaling y leaves the logits unchanged up to the eps term."""
    o = tiny_oracle()
    d = o.m.d_model
    W, g = o.W("lm_head"), o.W("final_norm")
    for a in (0.37, -2.5):
        np.testing.assert_allclose(o.lm_head(np.full((1, d), a)), np.sign(a) * (W @ g)[None, :], rtol=1e-5)
    y = rng.standard_normal((4, d))
    np.testing.assert_allclose(o.lm_head(7.0 * y), o.lm_head(y), rtol=1e-5, atol=1e-8)


def test_block_context_holds_the_committed_tokens():
    """Block mode: the first step of block 2 sees a context equal to a
    one-pass prefill of the prompt followed by block 1's final tokens (its
    logits rebuilt from a fresh session), so the committed rows are the
    block's tokens in their own order."""
    o = tiny_oracle(n_shared=1)
    logs = {}
    prompts, out = _gen(o, K=2, block_len=4, G=8, T=4,
                        hook=lambda b, n, z, r: logs.setdefault((b, n), (z.copy(), r["logits"])))
    z10, l10 = logs[(1, 0)]
    P = prompts.shape[1]
    o2 = O.Oracle(o.m, o._raw)
    sess = o2.new_session(2)
    o2.prefill(sess, out[:, :P + 4])
    cache = o2.anchor_forward(sess, z10)
    np.testing.assert_allclose(o2.denoise_logits(sess, z10, cache), l10, rtol=1e-10, atol=1e-12)


def test_encoder_pass_is_S_A_fusion_D():
    """The block-mode encoder pass (prefill / commit, App. C.1) runs the
    whole network causally: S, A, the fusion of (c, A(c)) and D, each layer
    keeping its K, V.  Rebuilt from the networks on a fresh session, layer by
    layer, its K and V are the session's."""
    for fusion in ("gated_mlp", "paired_attn"):
        o = tiny_oracle(n_shared=1, fusion=fusion)
        z = rng.integers(0, 63, size=9).astype(np.int32)
        s1 = o.new_session(1)[0]
        o._fresh_pass(s1, z)
        s2 = o.new_session(1)[0]
        pos = np.arange(9)
        c = o.S(z, pos, s2, causal=True, keep_kv=True)
        h = o.A(c, pos, s2, causal=True, keep_kv=True)
        ht = o.fuse(c, o.make_cache(c, h))
        o.D_hidden(ht, pos, s2, causal=True, keep_kv=True)
        assert sorted(s1.kv) == sorted(s2.kv) and any(k.startswith("denoise.") for k in s1.kv)
        for name in s1.kv:
            np.testing.assert_allclose(s1.kv[name][0], s2.kv[name][0], rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(s1.kv[name][1], s2.kv[name][1], rtol=1e-12, atol=1e-14)


# --------------------------------------------------------------------------- Gemma-3 layer details
def test_window_attention_brute_force_and_library():
    """Sliding-window attention (the local layers): a key at position j is
    visible to a query at position p iff p - j < W (and j <= p when causal).
    Checked against scalar loops with that rule written out, and against
    torch's SDPA with the same boolean mask."""
    Hq, Hkv, Lq, Lk, hd = 2, 1, 4, 9, 4
    q = rng.standard_normal((Hq, Lq, hd))
    k = rng.standard_normal((Hkv, Lk, hd))
    v = rng.standard_normal((Hkv, Lk, hd))
    qp, kp = np.array([5, 6, 7, 8]), np.arange(Lk)
    for causal in (False, True):
        for W in (1, 2, 3, 6):
            out = O.attention(q, k, v, qp, kp, causal, window=W)
            vis = [[(not causal or kp[j] <= qp[i]) and qp[i] - kp[j] < W for j in range(Lk)] for i in range(Lq)]
            for h in range(Hq):
                for i in range(Lq):
                    w = [math.exp(sum(q[h, i, t] * k[0, j, t] for t in range(hd)) / 2.0) if vis[i][j] else 0.0
                         for j in range(Lk)]
                    for t in range(hd):
                        assert abs(out[h, i, t] - sum(w[j] * v[0, j, t] for j in range(Lk)) / sum(w)) < 1e-12
            mask = torch.from_numpy(np.array(vis))
            ref = Fn.scaled_dot_product_attention(torch.from_numpy(q), torch.from_numpy(k).repeat(Hq, 1, 1),
                                                  torch.from_numpy(v).repeat(Hq, 1, 1), attn_mask=mask)
            np.testing.assert_allclose(out, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_window_special_cases():
    """A window at least as long as every query-key distance is no window; a
    window of 1 with causal attention leaves each query only its own key, so
    the output is that position's value."""
    Hq, Hkv, L, hd = 4, 2, 7, 8
    q = rng.standard_normal((Hq, L, hd))
    k = rng.standard_normal((Hkv, L, hd))
    v = rng.standard_normal((Hkv, L, hd))
    pos = np.arange(L) + 11
    for causal in (False, True):
        np.testing.assert_allclose(O.attention(q, k, v, pos, pos, causal, window=L),
                                   O.attention(q, k, v, pos, pos, causal), rtol=0, atol=0)
    own = O.attention(q, k, v, pos, pos, True, window=1)
    np.testing.assert_allclose(own, np.repeat(v, Hq // Hkv, axis=0), rtol=1e-14, atol=1e-14)
    # a non-causal window looks ahead without bound and back by less than W
    out = O.attention(q, k, v, pos, pos, False, window=1)
    last = O.attention(q[:, -1:], k, v, pos[-1:], pos, False, window=1)
    np.testing.assert_allclose(out[:, -1:], last, rtol=1e-14, atol=1e-14)
    np.testing.assert_allclose(last[:, 0], np.repeat(v, Hq // Hkv, axis=0)[:, -1], rtol=1e-14, atol=1e-14)


def test_gemma3_layer_pattern():
    """Five local layers per global one over the whole backbone (S, A, D):
    with 2 + 54 + 6 layers and global_every 6 the global layers are 5, 11,
    ..., 59; local layers take the window and the local RoPE base, global
    ones no window and the global base."""
    m = wl.POSTTRAIN_G3
    o = O.Oracle(m, {})
    names = ([f"shared.{i}." for i in range(m.n_shared)] + [f"anchor.{i}." for i in range(m.n_anchor)] +
             [f"denoise.{i}." for i in range(m.n_denoise)])
    assert [o.layer_index(n) for n in names] == list(range(62))
    kinds = [o.layer_kind(n) for n in names]
    assert [i for i, kd in enumerate(kinds) if kd[0] == 0] == [5, 11, 17, 23, 29, 35, 41, 47, 53, 59]
    assert {kd for kd in kinds} == {(1024, 1e4), (0, 1e6)}
    assert O.Oracle(wl.POSTTRAIN, {}).layer_kind("anchor.3.") == (0, 1e4)     # no pattern: all global


def _g3_oracle(eps=1e-6, **kw):
    base = dict(qk_norm=True, sandwich_norm=True, sliding_window=3, global_every=2, rope_theta_global=5e5,
                norm_eps=eps, n_shared=1)
    base.update(kw)
    return tiny_oracle(**base)


def test_qk_norm_removes_the_scale_of_q_and_k():
    """With QK-norm (and eps 0) scaling the Q or K rows of W_qkv by a positive
    constant leaves the layer unchanged; without it the output moves."""
    for qk in (True, False):
        o = _g3_oracle(eps=0.0, qk_norm=qk)
        m = o.m
        x = rng.standard_normal((6, m.d_model))
        ref = o.layer("anchor.0.", x, np.arange(6), None, False, False)
        w = dict(o._raw)
        wqkv = o.W("anchor.0.wqkv").copy()
        nq = m.n_heads * m.head_dim
        wqkv[:nq] *= 4.0            # powers of two: the float32 copy stays exact
        wqkv[nq:nq + m.n_kv_heads * m.head_dim] *= 0.5
        w["anchor.0.wqkv"] = wqkv.astype(np.float32)
        got = O.Oracle(m, w).layer("anchor.0.", x, np.arange(6), None, False, False)
        if qk:
            np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-11)
        else:
            assert not np.allclose(got, ref, rtol=1e-3)


def test_qk_norm_comes_before_rope():
    """RoPE keeps attention relative (a common position shift changes
    nothing) only if the per-dimension QK-norm gains act before the rotation;
    the gains here are far from uniform."""
    o = _g3_oracle(affine_std=0.5, sliding_window=0)
    x = rng.standard_normal((6, o.m.d_model))
    for name in ("anchor.0.", "anchor.1."):        # a local and a global layer
        a = o.layer(name, x, np.arange(6), None, False, False)
        b = o.layer(name, x, np.arange(6) + 29, None, False, False)
        np.testing.assert_allclose(a, b, rtol=1e-10, atol=1e-10)


def test_sandwich_norms():
    """Sandwich norms: zero post-norm gains silence both sub-blocks (the layer
    is the identity), and with eps 0 scaling W_o or W_down by a positive
    constant leaves the layer unchanged."""
    o = _g3_oracle(eps=0.0)
    m = o.m
    x = rng.standard_normal((5, m.d_model))
    w = dict(o._raw)
    w["anchor.0.post_attn_norm"] = np.zeros(m.d_model, np.float32)
    w["anchor.0.post_ffn_norm"] = np.zeros(m.d_model, np.float32)
    np.testing.assert_array_equal(O.Oracle(m, w).layer("anchor.0.", x, np.arange(5), None, False, False), x)
    ref = o.layer("anchor.0.", x, np.arange(5), None, False, False)
    w = dict(o._raw)
    w["anchor.0.wo"] = (o.W("anchor.0.wo") * 8.0).astype(np.float32)
    w["anchor.0.wdown"] = (o.W("anchor.0.wdown") * 0.125).astype(np.float32)
    np.testing.assert_allclose(O.Oracle(m, w).layer("anchor.0.", x, np.arange(5), None, False, False), ref,
                               rtol=1e-11, atol=1e-11)
    # only the attention branch silenced: x + RMSNorm(FFN(RMSNorm(x))) has unit-RMS increments
    w = dict(o._raw)
    w["anchor.0.post_attn_norm"] = np.zeros(m.d_model, np.float32)
    got = O.Oracle(m, w).layer("anchor.0.", x, np.arange(5), None, False, False)
    inc = (got - x) / o.W("anchor.0.post_ffn_norm")
    np.testing.assert_allclose(np.sqrt(np.mean(inc * inc, axis=-1)), 1.0, rtol=1e-12)


def test_global_layers_take_the_global_rope_base():
    """A backbone whose layers are all global with base rope_theta_global
    equals one without the pattern whose base is that value; the local
    layers of a patterned backbone use rope_theta."""
    a = _g3_oracle(global_every=1, sliding_window=2, rope_theta=1e4, rope_theta_global=5e5)
    b = O.Oracle(tiny_model(**{**a.m.__dict__, "global_every": 0, "sliding_window": 0, "rope_theta": 5e5,
                              "rope_theta_global": 0.0}), a._raw)
    x = rng.standard_normal((6, a.m.d_model))
    for name in ("shared.0.", "anchor.1."):
        np.testing.assert_allclose(a.layer(name, x, np.arange(6) + 3, None, True, False),
                                   b.layer(name, x, np.arange(6) + 3, None, True, False), rtol=0, atol=0)
    c = _g3_oracle(global_every=2, sliding_window=6)   # anchor.0 is layer 1: global; shared.0 is layer 0: local
    d = O.Oracle(tiny_model(**{**c.m.__dict__, "global_every": 0, "sliding_window": 0,
                              "rope_theta_global": 0.0}), c._raw)
    np.testing.assert_allclose(c.layer("shared.0.", x, np.arange(6), None, True, False),
                               d.layer("shared.0.", x, np.arange(6), None, True, False), rtol=0, atol=0)
    assert not np.allclose(c.layer("anchor.0.", x, np.arange(6), None, True, False),
                           d.layer("anchor.0.", x, np.arange(6), None, True, False))


def test_window_over_the_kv_context_equals_one_causal_pass():
    """Block mode with local layers: prefill + commit through the KV cache
    equals one causal pass over the concatenated rows, the window counting
    positions across the committed context."""
    o = _g3_oracle(sliding_window=3)
    z = rng.integers(0, 63, size=11).astype(np.int32)
    s1 = o.new_session(1)[0]
    o._fresh_pass(s1, z[:7])
    o._fresh_pass(s1, z[7:])
    s2 = o.new_session(1)[0]
    o._fresh_pass(s2, z)
    for name in s1.kv:
        np.testing.assert_allclose(s1.kv[name][0], s2.kv[name][0], rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(s1.kv[name][1], s2.kv[name][1], rtol=1e-10, atol=1e-12)
    # and the window changes the result (it is not silently ignored)
    s3 = O.Oracle(tiny_model(**{**o.m.__dict__, "sliding_window": 0}), o._raw).new_session(1)[0]
    O.Oracle(tiny_model(**{**o.m.__dict__, "sliding_window": 0}), o._raw)._fresh_pass(s3, z)
    assert not np.allclose(s3.kv["anchor.1."][0], s2.kv["anchor.1."][0])


def test_qk_norm_gains_belong_to_their_heads():
    """Zero Q-norm gains (with non-zero K-norm gains) zero every query and
    make attention uniform over the visible keys, exactly like zero Q rows of
    W_qkv; zero K-norm gains do the same as zero K rows.  A swap of the two
    gain vectors breaks both equalities."""
    o = _g3_oracle(affine_std=0.5, sandwich_norm=False)
    m = o.m
    nq, nk = m.n_heads * m.head_dim, m.n_kv_heads * m.head_dim
    x = rng.standard_normal((6, m.d_model))
    for gain, rows in (("q_norm", slice(0, nq)), ("k_norm", slice(nq, nq + nk))):
        a = dict(o._raw)
        a["anchor.0." + gain] = np.zeros(m.head_dim, np.float32)
        b = dict(o._raw)
        wqkv = o.W("anchor.0.wqkv").copy()
        wqkv[rows] = 0.0
        b["anchor.0.wqkv"] = wqkv.astype(np.float32)
        ya = O.Oracle(m, a).layer("anchor.0.", x, np.arange(6), None, False, False)
        yb = O.Oracle(m, b).layer("anchor.0.", x, np.arange(6), None, False, False)
        np.testing.assert_allclose(ya, yb, rtol=1e-12, atol=1e-12)
        assert not np.allclose(ya, o.layer("anchor.0.", x, np.arange(6), None, False, False))
