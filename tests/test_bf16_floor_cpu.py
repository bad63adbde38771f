"""Pins of the bf16-operand emulation in tests/bf16_floor.py (CPU), which the
GPU tests' agreement floor and depth gate are measured with: its rounding is
round-to-nearest-even bf16, and with every rounding site kept exact its
re-implemented layer, attention, fusion and head steps reproduce the fp64
oracle, so the only difference it measures is the rounding itself."""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)

import bf16_floor as F  # noqa: E402
import workloads as wl  # noqa: E402
from oracle import tadm_oracle as O  # noqa: E402

# every site the emulation rounds: backbone, gated-MLP fusion, head, paired-attention fusion
ALL_SITES = F.SITES + ("pa_in", "pa_j", "pa_qkv", "pa_p", "pa_o", "pa_r", "pa_hid", "pa_f", "pa_m")


def test_to_bf16_rounds_to_nearest_even():
    one = 1.0
    ulp = 2.0 ** -7                       # bf16 spacing in [1, 2)
    cases = {
        one: one,
        one + ulp / 2: one,               # tie: to the even mantissa (1.0)
        one + 3 * ulp / 2: one + 2 * ulp,  # tie: to the even mantissa (1 + 2 ulp)
        one + ulp / 2 + 2.0 ** -20: one + ulp,   # just above the tie
        one + ulp / 2 - 2.0 ** -20: one,         # just below the tie
        -(one + 3 * ulp / 2): -(one + 2 * ulp),
        0.0: 0.0,
        3.0e38: 2.0 ** 127 * 1.765625,    # large finite value rounds within range
    }
    x = np.array(list(cases), dtype=np.float64)
    got = F.to_bf16(x)
    assert np.array_equal(got, np.array(list(cases.values()))), got
    # every result is a bf16 value: its fp32 bit pattern has 16 zero low bits
    r = F.to_bf16(np.random.default_rng(0).standard_normal(4096) * 10.0 ** np.random.default_rng(1).integers(-6, 6, 4096))
    assert np.all((r.astype(np.float32).view(np.uint32) & 0xFFFF) == 0)


def test_to_bf16_matches_a_library_conversion():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    x = (rng.standard_normal(20000) * 10.0 ** rng.integers(-8, 8, 20000)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(F.to_bf16(x), ref)


def _single_block_logits(cls, m, host, B=2, R=48, seed=4):
    w = wl.Workload("t", m, batch=B, prompt_len=8, gen_len=R - 8, steps_per_block=8, K=2)
    z0 = wl.random_canvas(w, B, R, 0.8, seed=seed, start=8)
    z1 = wl.random_canvas(w, B, R, 0.5, seed=seed + 1, start=8)
    o = cls(m, host)
    s = o.new_session(B)
    cache = o.anchor_forward(s, z0)
    return o.denoise_logits(s, z1, cache)


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


MODELS = {
    "gated_mlp": dict(vocab=512, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32, ffn=256, n_shared=1,
                      n_anchor=2, n_denoise=1, dtype="bf16"),
    "paired_attn": dict(vocab=512, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32, ffn=256, n_shared=1,
                        n_anchor=2, n_denoise=1, dtype="bf16", fusion="paired_attn", fusion_rank=64,
                        fusion_heads=2, glu="geglu", tied_lm_head=True),
    "gemma3": dict(vocab=512, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32, ffn=256, n_shared=1,
                   n_anchor=3, n_denoise=2, dtype="bf16", sliding_window=12, qk_norm=True, sandwich_norm=True,
                   global_every=3, rope_theta_global=1e6),
}


@pytest.mark.parametrize("kind", list(MODELS))
def test_every_site_exact_reproduces_the_oracle(kind):
    m = wl.ModelConfig(**MODELS[kind])
    host = wl.make_weights(m, seed=2, affine_std=0.05)
    ref = _single_block_logits(O.Oracle, m, host)
    emu = _single_block_logits(F.with_exact(ALL_SITES), m, host)
    assert _rel(emu, ref) < 1e-12, _rel(emu, ref)


def test_every_site_exact_reproduces_the_oracle_in_block_mode():
    """Prompt prefill (KV context kept), a refresh and a stale step on the
    next block, with the Gemma-3 window cutting into the context."""
    m = wl.ModelConfig(**MODELS["gemma3"])
    host = wl.make_weights(m, seed=5, affine_std=0.05)
    out = F.block_step_case(m, host, batch=2, prompt_len=24, block_len=16, seed=6, T=4, exact=ALL_SITES)
    assert out["rel_l2"] < 1e-12, out["rel_l2"]


@pytest.mark.parametrize("site", ["head_in", "qkv_in", "p"])
def test_one_rounded_site_is_a_bf16_sized_perturbation(site):
    """Rounding a single site (the rest exact) changes the logits by about the
    bf16 unit roundoff (2^-9 relative), neither not at all nor grossly."""
    m = wl.ModelConfig(**MODELS["gated_mlp"])
    host = wl.make_weights(m, seed=2, affine_std=0.05)
    ref = _single_block_logits(O.Oracle, m, host)
    emu = _single_block_logits(F.with_exact(tuple(s for s in ALL_SITES if s != site)), m, host)
    assert 1e-5 < _rel(emu, ref) < 2e-2, _rel(emu, ref)
