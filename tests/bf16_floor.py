"""Token-agreement floor of an ideal bf16 tensor-core path (test infrastructure).

A bf16 tensor-core implementation must round every GEMM / attention operand
to bf16: the normalised activations entering the QKV, gate/up and output-head
GEMMs, Q, K and V after RoPE, the softmax numerators P, the attention output,
the GLU product and the fusion MLP's inputs (App. C.2).  Everything else
(accumulation, residual stream, norms, softmax sums) can stay exact.  This
script runs the oracle's arithmetic with exactly those roundings added (an
``Oracle`` subclass; weights, sampler and loop are the oracle's) through the
teacher-forced agreement protocol of the GPU model tests, with the fp64
oracle as the teacher, and writes the agreement it reaches to
``tests/golden/bf16_floor_small.json``.

That number is the floor of the protocol: no bf16 path, however exact its
accumulation, does better except by luck of rounding, because on random-init
weights the last masked positions of a block have near-tied top-2 logits and
a rounding of relative size 2^-9 flips some of them.  The GPU test compares
its own agreement with it.

Run (about 40 minutes of CPU):  python tests/bf16_floor.py
"""
from __future__ import annotations

import json
import math
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))

import workloads as wl  # noqa: E402
from oracle import tadm_oracle as O  # noqa: E402

# the agreement protocol of test_committed_token_agreement_teacher_forced[small_workload_dims]
PROTOCOL = dict(workload="small", batch=8, prompt_len=64, gen_len=192, steps=32, K=4, weight_seed=7,
                affine_std=0.0, prompt_seed=17)


def to_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 value (ties to even), returned as float64.
    Goes through float32 first, as the GPU's fp32 accumulators do."""
    a = np.ascontiguousarray(x, dtype=np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    rounded = ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) << 16
    return rounded.astype(np.uint32).view(np.float32).astype(np.float64)


# The tensor-core operand sites of the path, in the order the data meets them.
SITES = ("qkv_in", "qkv", "p", "o_in", "ffn_in", "down_in", "fusion_u", "fusion_hid", "head_in")


class Bf16Oracle(O.Oracle):
    """The oracle with bf16 operands at every tensor-core input, except the
    sites named in ``exact`` ("site" everywhere, "site@net" in one network:
    shared, anchor or denoise), which keep the oracle's arithmetic."""

    exact = frozenset()

    def _r(self, site, x):
        if site in self.exact or f"{site}@{self._net}" in self.exact:
            return x
        return to_bf16(x)

    def layer(self, name, x, pos, seq, causal, keep_kv):
        assert seq is None or not seq.kv, "single-block protocol only"
        self._net = name.split(".")[0]
        r = self._r
        m = self.m
        hd, Hq, Hkv, F = m.head_dim, m.n_heads, m.n_kv_heads, m.ffn
        L = x.shape[0]
        n = r("qkv_in", O.rms_norm(x, self.W(name + "attn_norm"), m.norm_eps))
        qkv = O.linear(n, self.W(name + "wqkv"))
        q = qkv[:, : Hq * hd].reshape(L, Hq, hd).transpose(1, 0, 2)
        k = qkv[:, Hq * hd: (Hq + Hkv) * hd].reshape(L, Hkv, hd).transpose(1, 0, 2)
        v = qkv[:, (Hq + Hkv) * hd:].reshape(L, Hkv, hd).transpose(1, 0, 2)
        q, k = O.rope(q, pos, m.rope_theta), O.rope(k, pos, m.rope_theta)
        q, k, v = r("qkv", q), r("qkv", k), r("qkv", v)
        group = Hq // Hkv
        o = np.empty_like(q)
        for h in range(Hq):
            # bf16 unnormalised numerators P; the row sums stay exact (fp32 on the GPU)
            s = q[h] @ k[h // group].T / math.sqrt(hd)
            if causal:
                s = np.where(pos[None, :] <= pos[:, None], s, O.NEG_INF)
            pe = np.exp(s - s.max(axis=-1, keepdims=True))
            o[h] = (r("p", pe) @ v[h // group]) / pe.sum(axis=-1, keepdims=True)
        x = x + O.linear(r("o_in", o.transpose(1, 0, 2).reshape(L, Hq * hd)), self.W(name + "wo"))
        n = r("ffn_in", O.rms_norm(x, self.W(name + "ffn_norm"), m.norm_eps))
        gu = O.linear(n, self.W(name + "wgu"))
        g, u = gu[:, :F], gu[:, F:]
        act = O.silu(g) if m.glu == "swiglu" else O.gelu_tanh(g)
        return x + O.linear(r("down_in", act * u), self.W(name + "wdown"))

    def fusion_gated_mlp(self, c, h):
        self._net = "fusion"
        r = self._r
        m, d, eps = self.m, self.m.d_model, self.m.norm_eps
        s = O.layer_norm(c, self.W("fusion.ln_c.w"), self.W("fusion.ln_c.b"), eps)
        a = O.layer_norm(h, self.W("fusion.ln_h.w"), self.W("fusion.ln_h.b"), eps)
        u = r("fusion_u", np.concatenate([s, a], axis=-1))
        wg1, bg1 = self.W("fusion.w_g1"), self.W("fusion.b_g1")
        g = O.sigmoid(O.linear(u, wg1[:d], bg1[:d]))
        hid = r("fusion_hid", O.gelu_erf(O.linear(u, wg1[d:], bg1[d:])))
        delta = O.linear(hid, self.W("fusion.w2"), self.W("fusion.b2"))
        return O.layer_norm(h + g * delta, self.W("fusion.ln_out.w"), self.W("fusion.ln_out.b"), eps)

    def lm_head(self, y):
        self._net = "head"
        n = self._r("head_in", O.rms_norm(y, self.W("final_norm"), self.m.norm_eps))
        return O.linear(n, self.W("embed") if self.m.tied_lm_head else self.W("lm_head"))


def with_exact(sites) -> type:
    """A Bf16Oracle subclass that keeps ``sites`` exact."""
    return type("Bf16OracleExact", (Bf16Oracle,), {"exact": frozenset(sites)})


def site_errors(p=PROTOCOL):
    """Logits rel-L2 against the fp64 oracle of one refresh + step on a
    partly unmasked canvas of the protocol's model (batch 2): with every site
    rounded ("all"), and with every site but one rounded ("all_but_<site>").
    The squared difference to "all" is that site's share of the error."""
    m = wl.get_workload(p["workload"]).model
    host = wl.make_weights(m, seed=p["weight_seed"], affine_std=p["affine_std"])
    B = 2
    w = wl.Workload("floor", m, batch=B, prompt_len=p["prompt_len"], gen_len=p["gen_len"],
                    steps_per_block=p["steps"], K=p["K"])
    z = wl.random_canvas(w, B, w.total_len, 0.3, seed=5, start=p["prompt_len"])
    ref = O.Oracle(m, host)
    s = ref.new_session(B)
    lr = ref.denoise_logits(s, z, ref.anchor_forward(s, z))
    out = {}
    for name, ex in [("all", ())] + [("all_but_" + t, (t,)) for t in SITES]:
        o = with_exact(ex)(m, host)
        ss = o.new_session(B)
        lg = o.denoise_logits(ss, z, o.anchor_forward(ss, z))
        out[name] = float(np.linalg.norm(lg - lr) / np.linalg.norm(lr))
    return out


def run(p=PROTOCOL, log=print, exact=()):
    m = wl.get_workload(p["workload"]).model
    assert m.fusion == "gated_mlp"
    host = wl.make_weights(m, seed=p["weight_seed"], affine_std=p["affine_std"])
    emu, ref = with_exact(exact)(m, host), O.Oracle(m, host)
    B, Tn, K, G = p["batch"], p["steps"], p["K"], p["gen_len"]
    w = wl.Workload("floor", m, batch=B, prompt_len=p["prompt_len"], gen_len=G, steps_per_block=Tn, K=K)
    z = wl.initial_canvas(w, wl.make_prompts(w, batch=B, seed=p["prompt_seed"]))
    s_emu, s_ref = emu.new_session(B), ref.new_session(B)
    n_sel = ok_sel = n_forced = ok_forced = n_masked = ok_masked = 0
    for n in range(Tn):
        if n % K == 0:
            c_emu, c_ref = emu.anchor_forward(s_emu, z), ref.anchor_forward(s_ref, z)
        g = emu.denoise_step(s_emu, z, c_emu, n, Tn, G)       # the bf16 path drives the canvas
        r = ref.denoise_step(s_ref, z, c_ref, n, Tn, G)       # the teacher sees the same canvas
        masked = z == m.mask_id
        committed = masked & (g["z"] != m.mask_id)
        ok = int((g["z"][committed] == r["tok"][committed]).sum())
        if O.unmask_count(n, Tn, G) >= int(masked.sum(axis=1).max()):
            n_forced += int(committed.sum())
            ok_forced += ok
        else:
            n_sel += int(committed.sum())
            ok_sel += ok
        n_masked += int(masked.sum())
        ok_masked += int((g["tok"][masked] == r["tok"][masked]).sum())
        log(f"step {n}: confidence-selected {ok_sel}/{n_sel}, all masked {ok_masked}/{n_masked}")
        z = g["z"]
    return dict(protocol=p, selected_ok=ok_sel, selected=n_sel, forced_ok=ok_forced, forced=n_forced,
                masked_ok=ok_masked, masked=n_masked)


if __name__ == "__main__":
    res = run()
    res["_source"] = ("written by tests/bf16_floor.py: the oracle with bf16 rounding at every tensor-core operand, "
                      "teacher-forced against the fp64 oracle")
    # where the flips come from: each site's share of the logits error, and the
    # agreement of the same protocol with the dominant site (the QKV
    # projections' input) kept exact, everywhere and in one network at a time
    res["site_logits_rel_l2"] = site_errors()
    for ex in (("qkv_in",), ("qkv_in@denoise",), ("qkv_in@anchor",)):
        r = run(log=lambda _: None, exact=ex)
        res["exact_" + "_".join(ex).replace("@", "_in_")] = {k: r[k] for k in
                                                             ("selected_ok", "selected", "forced_ok", "forced",
                                                              "masked_ok", "masked")}
    with open(os.path.join(HERE, "golden", "bf16_floor_small.json"), "w") as f:
        json.dump(res, f, indent=1)
        f.write("\n")
    print(json.dumps(res))
